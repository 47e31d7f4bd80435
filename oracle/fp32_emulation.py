"""fp32 emulation of the oracle's forward: the same steps in the same order, in
fp32 arithmetic instead of fp64.

TEST INFRASTRUCTURE, like the rest of this package: only the tests, the smoke
check, the bench's CPU leg and the script under tests/golden/ that writes the
stored tolerance bars may use it.  It shares no code with the CUDA path.

Why it exists.  On the reduced-precision configs the paper's recipe (Sec. 3.5:
16-bit projection operands, fp32 accumulation and recurrence) rounds every
operand of the per-hit matrix products to 16 bits.  Two correct implementations
that accumulate in different precisions (fp64 here, fp32 on the GPU) round a few
operands to different neighbouring 16-bit values, and the random-init network
amplifies those flips.  The spread between this emulation and the fp64 oracle
on the same inputs is therefore the error a correct fp32-accumulating
implementation is expected to show; the GPU parity bars for bf16 operands are
derived from it (tests/golden/make_bf16_bars.py).

Arithmetic: hit features normalised and featurised in fp64 then rounded to fp32
(the GPU forms the Fourier argument without rounding error); every product,
bias, gate, norm, scan step, residual, pooling sum and head operation in fp32
(numpy float32; matmul accumulates in fp32); the 16-bit operand rounding of the
oracle (round to nearest even) applied to the same operands.
"""
from __future__ import annotations

from typing import Optional

import numpy as np

from . import trackfit_oracle as O

F32 = np.float32


def _op(x, prec):
    """Operand of a per-hit product, rounded to bf16 (1) or fp16 (2); fp32 result.
    Both formats embed exactly in fp32, so the round trip through fp64 is exact."""
    x = np.asarray(x, dtype=F32)
    if prec == 1:
        return O.bf16_round(x.astype(np.float64)).astype(F32)
    if prec == 2:
        return O.fp16_round(x.astype(np.float64)).astype(F32)
    return x


# Accumulation order of the fp32 matrix products: "k16" = the K axis in
# consecutive blocks of 16 products, each block summed and added to a running
# fp32 accumulator (the step of one tensor-core instruction), rounding to
# nearest; "k16rz" = the same steps with each new accumulator value rounded
# toward zero, and the accumulation onto x' (the second MLP product) with the
# tensor core's truncation of every product (_tc_onto); "blas" (not in ORDERS) =
# numpy's float32 matmul as it blocks it.  All are fp32 accumulations of the
# same product; "k16rz" is the rounding a tensor core applies (measured: its fp32
# sums of same-sign products fall short of the exact sum by a few ulps, and by
# tens of ulps when added onto a large accumulator, a bias round-to-nearest does
# not have), and a systematically shortened accumulator moves more 16-bit
# roundings across a boundary than an unbiased one.  Their spread against the
# fp64 oracle is what the tolerance covers.
ORDERS = ("k16", "k16rz")


def _tc_onto(acc, a, bt):
    """acc + a @ bt in steps of 16 products with the tensor core's truncation: each
    exact product is truncated toward zero to a quarter of the fp32 ulp of the
    largest magnitude among the step's products and the accumulator, the step's sum
    (exact) is added to the accumulator and the result rounded toward zero.  This
    reproduces the measured statistics of tcgen05 fp32 accumulation exactly for
    same-sign products and for products added onto a large accumulator (the case
    where truncation matters: MLP2 accumulating onto x').  torch CPU operations for
    speed; every value is exact in fp64 until the final rounding."""
    import torch
    A = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64))
    Bt = torch.from_numpy(np.ascontiguousarray(bt, dtype=np.float64))
    out = np.empty(acc.shape, dtype=F32)
    for r0 in range(0, A.shape[0], 512):
        ac = torch.from_numpy(np.ascontiguousarray(acc[r0:r0 + 512], dtype=np.float64))
        for k0 in range(0, A.shape[1], 16):
            P = A[r0:r0 + 512, k0:k0 + 16, None] * Bt[None, k0:k0 + 16, :]         # exact (16-bit operands)
            m = torch.maximum(ac.abs(), P.abs().amax(dim=1))
            e = torch.frexp(torch.where(m > 0, m, torch.ones_like(m)))[1]        # m = f 2^e, f in [0.5, 1)
            q = torch.ldexp(torch.ones_like(m), e - 26)[:, None, :]             # 2^(floor(log2 m) - 25)
            s64 = ac + (torch.trunc(P / q) * q).sum(dim=1)
            f = s64.to(torch.float32)
            over = f.to(torch.float64).abs() > s64.abs()
            f = torch.where(over, torch.nextafter(f, torch.zeros_like(f)), f)
            ac = f.to(torch.float64)
        out[r0:r0 + 512] = ac.to(torch.float32).numpy()
    return out


def _add_toward_zero(acc, blk):
    """acc + blk (fp32 arrays) rounded toward zero: the round-to-nearest sum, moved
    one step toward zero where it rounded away from it (the exact rounding error
    of the sum, from Knuth's TwoSum, has the opposite sign).  One step toward zero
    is one less in the magnitude bits of the float."""
    s = acc + blk
    bb = s - acc
    err = acc - (s - bb)
    err += blk - bb
    away = (err < 0) & (s > 0)
    away |= (err > 0) & (s < 0)
    s.view(np.int32)[...] -= away
    return s


def _matmul(a, bt, order, init=None):
    """a @ bt accumulated in fp32 in the given order; init (same shape as the
    result, the blocked orders only) is the accumulator's starting value."""
    if order == "blas":
        return (a @ bt).astype(F32)
    if order == "seq":
        # one product at a time, fused multiply-add rounding to nearest (the
        # CUDA-core path's order): exact product plus accumulator, rounded once
        acc = np.zeros(a.shape[:-1] + (bt.shape[1],), dtype=F32) if init is None else init.astype(F32)
        for k in range(a.shape[-1]):
            acc = (acc.astype(np.float64) + a[..., k:k + 1].astype(np.float64) * bt[k].astype(np.float64)).astype(F32)
        return acc
    if order not in ("k16", "k16rz"):
        raise ValueError(order)
    shape = a.shape[:-1] + (bt.shape[1],)
    a2 = a.reshape(-1, a.shape[-1])
    out = np.empty((a2.shape[0], bt.shape[1]), dtype=F32)
    init2 = None if init is None else init.reshape(-1, bt.shape[1])
    for r0 in range(0, a2.shape[0], 2048):           # rows in chunks: bounded temporaries
        ac = np.ascontiguousarray(a2[r0:r0 + 2048])
        acc = np.zeros((ac.shape[0], bt.shape[1]), dtype=F32) if init2 is None else init2[r0:r0 + 2048].astype(F32)
        for k0 in range(0, a.shape[-1], 16):
            blk = (ac[:, k0:k0 + 16] @ bt[k0:k0 + 16]).astype(F32)
            acc = (acc + blk).astype(F32) if order == "k16" else _add_toward_zero(acc, blk)
        out[r0:r0 + 2048] = acc
    return out.reshape(shape)


def _lin(x, w, b, prec, order="k16", rows=None, onto=None):
    """x W^T + b over the last axis of x; with rows (a boolean mask over x's
    leading axes) only those rows are computed, the others are zero (padding
    rows, whose values never reach a result).  onto (blocked orders): the
    accumulation starts from it, giving onto + x W^T + b."""
    if order == "blas" and onto is not None:
        return (onto + _lin(x, w, b, prec, order, rows)).astype(F32)
    if order == "k16rz" and onto is not None:
        xr = x if rows is None else x[rows]
        base = onto if rows is None else onto[rows]
        res = (_tc_onto(base.reshape(-1, base.shape[-1]), _op(xr, prec).reshape(-1, xr.shape[-1]), _op(w, prec).T)
               .reshape(base.shape) + b.astype(F32)).astype(F32)
        if rows is None:
            return res
        out = np.zeros(x.shape[:-1] + (w.shape[0],), dtype=F32)
        out[rows] = res
        return out
    if rows is None:
        return (_matmul(_op(x, prec), _op(w, prec).T, order, onto) + b.astype(F32)).astype(F32)
    out = np.zeros(x.shape[:-1] + (w.shape[0],), dtype=F32)
    out[rows] = (_matmul(_op(x[rows], prec), _op(w, prec).T, order, None if onto is None else onto[rows])
                 + b.astype(F32)).astype(F32)
    return out


def fourier(u, scales):
    """The oracle's Fourier features as an fp32 evaluation computes them: the
    argument s_k u reduced modulo 2 into [-1, 1] (exactly, in fp64), rounded to
    fp32, then sin and cos of pi times that fp32 argument, rounded to fp32.  The
    argument's rounding (a relative 6e-8) is the one that matters: near a zero
    of the sine it moves the value by far more than the sine's own rounding, and
    so across 16-bit rounding boundaries of the embedding's operand."""
    s = np.asarray(scales, dtype=np.float64)
    a = np.asarray(u, dtype=np.float64)[..., :, None] * s
    a = (a - 2.0 * np.rint(0.5 * a)).astype(F32).astype(np.float64)
    e = np.concatenate([np.sin(np.pi * a), np.cos(np.pi * a)], axis=-1).astype(F32)
    return e.reshape(np.shape(u)[:-1] + (2 * np.shape(u)[-1] * s.size,))


def sigmoid(x):
    with np.errstate(over="ignore"):
        return (F32(1.0) / (F32(1.0) + np.exp(-x, dtype=F32))).astype(F32)


def silu(x):
    return (x * sigmoid(x)).astype(F32)


def rmsnorm(x, g, eps):
    ms = np.mean(x * x, axis=-1, keepdims=True, dtype=F32)
    return (x / np.sqrt(ms + F32(eps)) * g.astype(F32)).astype(F32)


def linear_scan(a, b, x, valid, reverse=False):
    """h_t = a_t h_{t-1} + b_t x_t along axis 1 in fp32 (masked as the oracle's)."""
    B, T, C = x.shape
    h = np.zeros((B, C), dtype=F32)
    out = np.zeros((B, T, C), dtype=F32)
    steps = range(T - 1, -1, -1) if reverse else range(T)
    for t in steps:
        v = valid[:, t, None]
        h = np.where(v, (a[:, t] * h + b[:, t] * x[:, t]).astype(F32), h)
        out[:, t] = np.where(v, h, F32(0.0))
    return out


def encoder_layer(x, W, l, cfg, valid, prec, order="k16"):
    """One layer, the oracle's encoder_layer in fp32 (mean-pooling form)."""
    D, H = cfg["d_model"], cfg["d_hidden"]
    p = f"layer{l}."
    xh = rmsnorm(x, W[p + "g"], cfg["rms_eps"])
    proj = _lin(xh, W[p + "w_in"], W[p + "b_in"], prec, order, valid)
    z_f = sigmoid(proj[..., 0:H])
    n_f = proj[..., H:2 * H]
    z_b = sigmoid(proj[..., 2 * H:3 * H])
    n_b = proj[..., 3 * H:4 * H]
    gate = sigmoid(proj[..., 4 * H:4 * H + D])
    one = F32(1.0)
    h_f = linear_scan((one - z_f).astype(F32), z_f, n_f, valid)
    h_b = linear_scan((one - z_b).astype(F32), z_b, n_b, valid, reverse=True)
    y = np.concatenate([h_f, h_b], axis=-1)
    m = _lin(y, W[p + "w_m"], W[p + "b_m"], prec, order, valid)
    x1 = (x + m * gate).astype(F32)
    u = silu(_lin(x1, W[p + "w1"], W[p + "b1"], prec, order, valid))
    # the second MLP product accumulates onto x' (the association the tensor-core
    # path uses: x' is the accumulator's starting value, the bias is added last)
    x2 = _lin(u, W[p + "w2"], W[p + "b2"], prec, order, valid, onto=x1)
    return np.where(valid[..., None], x2, F32(0.0)), h_f, h_b


def forward(cfg: dict, blob, hits, n_hits, capture: Optional[dict] = None, order: str = "k16"):
    """Track parameters [B, 5] (returned as fp64 holding fp32 values) for mean
    pooling; with capture, also the pooled vector after every layer
    (capture["pooled_by_layer"][l], fp64 holding fp32 values)."""
    if int(cfg["pool"]) != 0:
        raise ValueError("the fp32 emulation covers mean pooling only")
    Wd = O.split_blob(cfg, blob)
    W = {k: v.astype(F32) for k, v in Wd.items()}
    prec = int(cfg["precision"])
    hits = np.asarray(hits)
    n_hits = np.asarray(n_hits).astype(np.int64)
    B, T, _ = hits.shape
    bad = (n_hits < 1) | (n_hits > T)
    n_ok = np.where(bad, 1, n_hits)
    valid = np.arange(T)[None, :] < n_ok[:, None]
    e = fourier(O.normalise(hits, cfg["feat_min"], cfg["feat_max"]), cfg["fourier_scale"])
    hdn = silu(_lin(e, W["emb.w1"], W["emb.b1"], prec, order, valid))
    x = np.where(valid[..., None], _lin(hdn, W["emb.w2"], W["emb.b2"], prec, order, valid), F32(0.0))
    nf = n_ok[:, None].astype(F32)
    by_layer = []
    for l in range(cfg["n_layers"]):
        x, _, _ = encoder_layer(x, W, l, cfg, valid, prec, order)
        if capture is not None:
            by_layer.append((np.sum(x, axis=1, dtype=F32) / nf).astype(np.float64))
    pv = (np.sum(x, axis=1, dtype=F32) / nf).astype(F32)
    hn = rmsnorm(pv, W["head.g"], cfg["rms_eps"])
    hid = silu((hn @ W["head.w1"].T + W["head.b1"]).astype(F32))
    q = (hid @ W["head.w2"].T + W["head.b2"]).astype(F32)
    nq = cfg["n_quantiles"]
    q = q.reshape(B, q.shape[1] // nq, nq)
    out = np.where(bad[:, None], np.nan, q[:, :, nq // 2].astype(np.float64))
    if capture is not None:
        capture.update(pooled=pv.astype(np.float64), pooled_by_layer=by_layer, quantiles=q.astype(np.float64))
    return out
