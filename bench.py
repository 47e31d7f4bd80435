"""Throughput benchmark of the track-fit encoder on GB300.

One step = one forward of the whole hot path (Fourier embedding, every minGRU
layer, pooling, head) over the full synthetic batch of the workload (default:
large, 1,048,576 tracks, d_model 256, 8 layers, bf16 operands).  Inputs are
resident in HBM when the timed region starts; the hit batch (503 MB) is larger
than L2, so no flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload large] [--impl ours|reference]
  python bench.py --sweep        # length sweep: T = 8/16/32/64 x batch 4k-1M, one line per point
  python bench.py --seed         # analytic fp64 seed + features + decode, and its share of the forward
  python bench.py --packed       # packed, unpadded input against the padded entry point
  python bench.py --paper        # the paper's model: seed, 15-feature encoder, decode per step
  python bench.py --transformer  # the same with the Transformer encoder of the encoder comparison

N > 1 runs under torch.distributed.run, one rank per GPU; every rank processes
its own full batch (replicas, weak scaling; the path has no exchange step).
--impl reference times the CPU oracle on bounded samples of the same workload
(rank 0 only).  Prints one JSON line.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_32479_gb300 import workloads as W  # noqa: E402

METRIC = "tracks/sec at 1 GB300 (device-timed) and % of HBM/tensor roofline vs CPU oracle"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
KERNEL_SRC = os.path.join(ROOT, "paper_2609_32479_gb300", "csrc", "tc_forward.cu")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "tc_forward_large.traffic.json")


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as fh:
            d = json.load(fh)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


def flops_per_hit(m: W.ModelConfig) -> int:
    """Algorithmic multiply-add work per valid hit: embedding 2(E D + D^2) plus, per
    layer, 2 D (4H + D) + 2 (2H) D + 2 (2 D^2) (= 24 D^2 at H = 1.5 D)."""
    D, H, E = m.d_model, m.d_hidden, m.embed_dim
    per_layer = 2 * D * (4 * H + D) + 2 * 2 * H * D + 4 * D * D
    return 2 * (E * D + D * D) + m.n_layers * per_layer


def flops_per_track_head(m: W.ModelConfig) -> int:
    return 2 * (m.pooled_dim * m.head_hidden + m.head_hidden * m.n_out)


def bytes_per_track(m: W.ModelConfig) -> int:
    """Compulsory HBM traffic of one track: padded hits in, hit count in, 5 outputs out."""
    return m.max_hits * 5 * 4 + 4 + 5 * 4


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.flush()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
                for n, v in zip(names, r[5:9]):
                    if v.strip().lower() == "active":
                        reasons.add(n)
            except (ValueError, IndexError):
                continue
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(mx)), "reasons": sorted(reasons),
                "samples": len(sm)}


def stratified_sample(n_hits: np.ndarray, n: int, seed: int = 7) -> np.ndarray:
    """n track indices covering every hit count present in proportion."""
    rng = np.random.default_rng(seed)
    idx = rng.choice(n_hits.size, size=min(n, n_hits.size), replace=False)
    extra = [int(np.nonzero(n_hits == k)[0][0]) for k in np.unique(n_hits)]
    return np.unique(np.concatenate([idx, extra]))


_ORACLE = {}


def _oracle_init(model, seed):
    """Worker set-up: the oracle and the workload's weights (regenerated from their
    seed rather than shipped to every worker)."""
    from oracle import trackfit_oracle as O
    _ORACLE["O"] = O
    _ORACLE["cfg"] = dataclasses.asdict(model)
    _ORACLE["blob"] = W.gen_weights(model, seed)


def _oracle_chunk(hits, n_hits):
    return _ORACLE["O"].forward(_ORACLE["cfg"], _ORACLE["blob"], hits, n_hits)


class OraclePool:
    """The CPU oracle, as it stands, run on every host core: one single-threaded
    process per core (BLAS limited to one thread each), tracks split into chunks.
    Started with spawn, so that no worker is forked from a process that has used
    the GPU."""

    def __init__(self, w: W.Workload):
        import concurrent.futures
        import multiprocessing
        self.workers = host_cores()
        keep = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
        for k in keep:
            os.environ[k] = "1"   # inherited by the spawned workers
        try:
            self.ex = concurrent.futures.ProcessPoolExecutor(
                max_workers=self.workers, mp_context=multiprocessing.get_context("spawn"),
                initializer=_oracle_init, initargs=(w.model, w.weight_seed))
            # every worker started and set up before anything is timed
            list(self.ex.map(_oracle_chunk, [np.zeros((1, w.model.max_hits, w.model.n_features), np.float32)] *
                             (2 * self.workers), [np.ones(1, np.int32)] * (2 * self.workers)))
        finally:
            for k, v in keep.items():
                if v is None:
                    os.environ.pop(k, None)
                else:
                    os.environ[k] = v

    def forward(self, hits, n_hits, chunk=64):
        parts = list(self.ex.map(_oracle_chunk, [hits[i:i + chunk] for i in range(0, len(n_hits), chunk)],
                                 [n_hits[i:i + chunk] for i in range(0, len(n_hits), chunk)]))
        return np.concatenate(parts)

    def close(self):
        self.ex.shutdown()


def run_oracle_sample(w: W.Workload, blob, tb, budget_s: float, pool: "OraclePool"):
    """Time the CPU oracle (as it stands, on every host core) on a bounded sample of
    about budget_s seconds: returns (tracks/s, sample indices, outputs, seconds)."""
    cal = stratified_sample(tb.n_hits, 16 * pool.workers, seed=1)
    t0 = time.perf_counter()
    pool.forward(tb.hits[cal], tb.n_hits[cal], chunk=16)
    per = (time.perf_counter() - t0) / len(cal)
    n = int(max(16, min(65536, budget_s / max(per, 1e-6))))
    idx = stratified_sample(tb.n_hits, n)
    t0 = time.perf_counter()
    out = pool.forward(tb.hits[idx], tb.n_hits[idx])
    dt = time.perf_counter() - t0
    return idx.size / dt, idx, out, dt


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def config_block(w: W.Workload, tb) -> dict:
    m = w.model
    hist = W.length_histogram(tb.n_hits)
    return {"workload": w.name, "n_tracks": w.n_tracks, "max_hits": m.max_hits, "d_model": m.d_model,
            "d_hidden": m.d_hidden, "n_layers": m.n_layers, "pool": "mean" if m.pool == 0 else "endpoints",
            "precision": {0: "fp32", 1: "bf16", 2: "fp16"}[m.precision],
            "mean_hits": float(tb.n_hits.mean()), "hit_histogram": hist,
            "l2": "inputs larger than L2 (hits %.0f MB > 129 MB); no flush" % (tb.hits.nbytes / 1e6),
            "parallelism": "replicas"}


def reference_main(args, w: W.Workload):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    budget = max(2.0, min(15.0, 150.0 / max(1, args.steps + args.warmup)))
    pool = OraclePool(w)
    for _ in range(args.warmup):
        run_oracle_sample(w, blob, tb, min(budget, 3.0), pool)
    vals, tot_t, tot_n = [], 0.0, 0
    for _ in range(args.steps):
        v, idx, _, dt = run_oracle_sample(w, blob, tb, budget, pool)
        vals.append(v)
        tot_t += dt
        tot_n += idx.size
    pool.close()
    value = tot_n / tot_t
    cores = pool.workers
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tracks/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_t / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config_block(w, tb),
            "cpu_baseline": {"value": value, "unit": "tracks/s", "cores": cores, "kind": "oracle",
                             "sample": f"{tot_n // args.steps} stratified tracks of {w.name} per step (numpy fp64, "
                                       f"one single-threaded oracle process per core)"},
            "e2e": {"value": value, "unit": "tracks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def parity_block(w: W.Workload, blob, tb, gpu_out, idx, ref, emul_max_tracks: int = 384) -> dict:
    """Per-track parity of the GPU output on the oracle's sample.  For 16-bit
    operands the fp32 emulation of the oracle (same arithmetic, fp32 accumulation)
    runs on the first tracks of the sample, giving the spread a correct
    fp32-accumulating implementation shows on the same tracks; the 2e-3 bar on
    every track is reported as its own pass/fail."""
    from tests.helpers import bf16_bars, track_errors
    e = track_errors(gpu_out[idx], ref)
    out = {"tracks": int(idx.size), "metric": "per track: max over the 5 outputs of |g - r| / max(|r|, column RMS)",
           "p90": float(np.percentile(e, 90)), "p99": float(np.percentile(e, 99)), "max": float(e.max()),
           "every_track_within_2e-3": bool(e.max() <= 2e-3)}
    if w.model.precision != W.PRECISION_FP32 and w.model.pool == W.POOL_MEAN:
        from oracle import fp32_emulation as E
        k = min(emul_max_tracks, idx.size)
        sub = idx[:k]
        ems = [E.forward(dataclasses.asdict(w.model), blob, tb.hits[sub], tb.n_hits[sub], order=o) for o in E.ORDERS]
        e_ems = [track_errors(em, ref[:k]) for em in ems]
        e_g = track_errors(gpu_out[sub], ref[:k])
        bmean, b90, bmx = bf16_bars(ref[:k], ems)
        out["same_tracks_vs_fp32_emulation"] = {
            "tracks": int(k), "gpu_mean": float(e_g.mean()), "gpu_p90": float(np.percentile(e_g, 90)),
            "gpu_max": float(e_g.max()), "orders": list(E.ORDERS),
            "emulation_mean": [float(x.mean()) for x in e_ems],
            "emulation_p90": [float(np.percentile(x, 90)) for x in e_ems],
            "emulation_max": [float(x.max()) for x in e_ems],
            "bar_mean": bmean, "bar_p90": b90, "bar_max": bmx,
            "gate_ok": bool(e_g.mean() <= bmean and np.percentile(e_g, 90) <= b90 and e_g.max() <= bmx)}
    return out


def sweep_main(args):
    """Throughput over the length sweep: for T in 8/16/32/64 (d_model 128, 6 layers,
    bf16 operands, every track T hits) and batches 4k-1M, one JSON line per point.
    Each timed forward is preceded by an L2 flush (a 256 MB write, outside the
    timed interval); per point the median of the timed forwards is reported."""
    import torch
    from paper_2609_32479_gb300 import trackfit as TF
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peaks, peak_kind = load_peaks()
    peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    for T in (8, 16, 32, 64):
        w = W.workload(f"sweep{T}")
        tb = W.gen_tracks(w)
        blob = W.gen_weights(w.model, w.weight_seed)
        m = w.model
        hits_all = torch.from_numpy(tb.hits).to(dev)
        n_all = torch.from_numpy(tb.n_hits).to(dev)
        with TF.Trackfit(m, blob) as tf:
            for B in W.SWEEP_BATCHES:
                hits, n_hits = hits_all[:B], n_all[:B]
                out = torch.empty((B, 5), dtype=torch.float32, device=dev)
                for _ in range(3):
                    tf.forward(hits, n_hits, out, stream)
                reps = max(5, min(50, int(2.0e7 // (B * T))))
                times = []
                tf.profile(True)
                tf.profile_read()
                for _ in range(reps):
                    flush.fill_(1.0)
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record(stream)
                    tf.forward(hits, n_hits, out, stream)
                    e1.record(stream)
                    torch.cuda.synchronize(dev)
                    times.append(e0.elapsed_time(e1))
                kern_ms, kern_n = tf.profile_read()
                tf.profile(False)
                st, nbad = tf.device_errors(stream)
                ms = float(np.median(times))
                flops = B * T * flops_per_hit(m) + B * flops_per_track_head(m)
                kms = kern_ms / max(kern_n, 1)
                line = {"metric": METRIC, "value": B / (ms * 1e-3), "unit": "tracks/s", "n_gpus": 1,
                        "steps": reps, "warmup": 3, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
                        "vs_baseline": None, "dtype": "bf16", "data": "synthetic helix tracks + random-init weights",
                        "config": {"workload": w.name, "n_tracks": B, "max_hits": T, "d_model": m.d_model,
                                   "n_layers": m.n_layers, "l2": "flushed (256 MB write) before every timed forward"},
                        "path": tf.path,
                        "roofline": {"bound": "tensor", "achieved": flops / (kms * 1e-3) / 1e12, "peak": peak,
                                     "unit": "TFLOP/s", "frac": flops / (kms * 1e-3) / 1e12 / peak,
                                     "peak_kind": f"{peak_kind} bf16 dense burst", "kernel_ms": kms,
                                     "step_frac": flops / (ms * 1e-3) / 1e12 / peak},
                        "device_errors": {"status": st, "bad_tracks": nbad}}
                print(json.dumps(line), flush=True)
        del hits_all, n_all
    return 0


def _time_events(fn, reps, stream):
    """Median milliseconds of fn() over reps runs, CUDA events on `stream`."""
    import torch
    ts = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    return float(np.median(ts))


def next_main(args, w: W.Workload):
    """--seed: the analytic fp64 seed with its per-hit features and the decode
    (Sec. 3.1, 3.3) over the workload's batch, with its share of seed + forward
    (the paper reports 9-12 %).  --packed: the packed, unpadded entry point
    (Sec. 3.5) against the padded one on the same tracks.  One JSON line each."""
    import torch
    from paper_2609_32479_gb300 import trackfit as TF
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    B, T = w.n_tracks, w.model.max_hits
    hits = torch.from_numpy(tb.hits).to(dev)
    nh = torch.from_numpy(tb.n_hits).to(dev)
    out = torch.empty((B, 5), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    reps = max(args.steps, 3)
    with TF.Trackfit(w.model, blob) as tf:
        for _ in range(max(args.warmup, 1)):
            tf.forward(hits, nh, out, stream)
        fwd_ms = _time_events(lambda: tf.forward(hits, nh, out, stream), reps, stream)
        base = {"n_gpus": 1, "steps": reps, "warmup": max(args.warmup, 1), "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "data": "synthetic helix tracks + random-init weights (seeded)",
                "path": tf.path}
        if args.seed:
            seed = torch.empty((B, 5), dtype=torch.float64, device=dev)
            feats = torch.empty((B, T, 3), dtype=torch.float32, device=dev)
            corr = torch.zeros((B, 5), dtype=torch.float32, device=dev)
            dec = torch.empty((B, 5), dtype=torch.float32, device=dev)

            def seed_step():
                TF.seed(hits, nh, w.b_field, seed, feats, stream)
                TF.decode(seed, corr, dec, stream)
            for _ in range(max(args.warmup, 1)):
                seed_step()
            ms = _time_events(seed_step, reps, stream)
            line = dict(base, metric="analytic fp64 seed + residual features + decode, tracks/sec (device-timed)",
                        value=B / (ms * 1e-3), unit="tracks/s", ms_per_step=ms, dtype="f64",
                        config={"workload": w.name, "n_tracks": B, "max_hits": T, "b_field_tesla": w.b_field,
                                "l2": "inputs larger than L2; no flush"},
                        seed_share_of_seed_plus_forward=ms / (ms + fwd_ms), forward_ms=fwd_ms,
                        seed_us_per_track=1e3 * ms / B)
        else:
            rows = [tb.hits[b, :tb.n_hits[b]] for b in range(B)]
            packed = torch.from_numpy(np.ascontiguousarray(np.concatenate(rows))).to(dev)
            offs = torch.from_numpy(np.concatenate([[0], np.cumsum(tb.n_hits)]).astype(np.int64)).to(dev)
            outp = torch.empty_like(out)
            for _ in range(max(args.warmup, 1)):
                tf.forward_packed(packed, offs, outp, stream)
            ms = _time_events(lambda: tf.forward_packed(packed, offs, outp, stream), reps, stream)
            torch.cuda.synchronize()
            same = bool(torch.equal(outp, out))
            line = dict(base, metric=METRIC + " (packed input)", value=B / (ms * 1e-3), unit="tracks/s",
                        ms_per_step=ms, dtype={0: "f32", 1: "bf16", 2: "f16"}[w.model.precision],
                        config={"workload": w.name, "n_tracks": B, "layout": "packed", "l2": "inputs larger than L2"},
                        padded_forward_ms=fwd_ms, matches_padded_bitwise=same,
                        input_bytes_per_track={"packed": float((packed.numel() * 4 + offs.numel() * 8) / B),
                                               "padded": float(T * 20 + 4)})
        print(json.dumps(line))
    return 0


# FP32 ALU peak of the CUDA-core path, from unit counts and clocks: 152 SMs x 128
# FP32 lanes x 2 flop per FMA x 2.07 GHz (the maximum SM clock) = 80.5 TFLOP/s.
FP32_ALU_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def encoder_flops(m, n_hits):
    """Algorithmic flops of the encoder over tracks with these hit counts: the
    per-hit products (embedding, then per layer the projections; for the
    Transformer also q.k and p.v over each track's hits) and the head."""
    D, H, E = m.d_model, m.d_hidden, m.embed_dim
    n = np.asarray(n_hits, dtype=np.int64)
    per_hit = 2 * (E * D + D * D)
    if m.topology == W.TOPOLOGY_ATTENTION:
        per_hit += m.n_layers * 2 * (3 * D * D + D * D + 2 * H * D)
        attn = m.n_layers * 4 * D * int((n * n).sum())
    else:
        per_hit += sum(2 * (D if l == 0 else 2 * H) * 4 * H for l in range(m.n_layers))
        attn = 0
    return int(n.sum()) * per_hit + attn + len(n) * flops_per_track_head(m)


def product_flops(m, n_hits):
    """Algorithmic flops of the per-hit matrix products alone (what the packed-row
    tensor-core kernel computes): the embedding and every layer's products over
    the valid hits."""
    D, H, E = m.d_model, m.d_hidden, m.embed_dim
    per_hit = 2 * (E * D + D * D)
    if m.topology == W.TOPOLOGY_ATTENTION:
        per_hit += m.n_layers * 2 * (3 * D * D + D * D + 2 * H * D)
    else:
        per_hit += sum(2 * (D if l == 0 else 2 * H) * 4 * H for l in range(m.n_layers))
    return int(np.asarray(n_hits, dtype=np.int64).sum()) * per_hit


def product_bytes(m, n_hits):
    """Algorithmic HBM bytes of the per-hit products over the valid hits: each
    product reads its 16-bit operand rows (and, with a residual, the fp32 stream)
    and writes its results (fp32 projections and residual stream, 16-bit operands
    of the next product); the weights stay in L2."""
    D, H, E = m.d_model, m.d_hidden, m.embed_dim
    per_hit = 2 * E + 2 * D                       # e1: Fourier operand in, SiLU operand out
    if m.topology == W.TOPOLOGY_ATTENTION:
        per_hit += 2 * D + 4 * D + 2 * D          # e2: x and its pre-norm operand
        for l in range(m.n_layers):
            last = l + 1 == m.n_layers
            per_hit += 2 * D + 4 * 3 * D          # q, k, v
            per_hit += 2 * D + 4 * D + 4 * D + 2 * D   # W_o: operand, residual in, x' and its pre-norm out
            per_hit += 2 * D + 2 * H              # W_1: SiLU operand out
            per_hit += 2 * H + 4 * D + 4 * D + (0 if last else 2 * D)   # W_2
    else:
        per_hit += 2 * D + 2 * D                  # e2: the first layer's operand
        for l in range(m.n_layers):
            per_hit += 2 * (D if l == 0 else 2 * H) + 4 * 4 * H
    return int(np.asarray(n_hits, dtype=np.int64).sum()) * per_hit


PAPER_CONTEXT = {"paper": "the paper reports 5.41 M tracks/s on one H100 NVL for its trained minGRU model on its data",
                 "transformer": "the paper reports 3.18 M tracks/s on one H100 NVL for its Transformer of the same "
                                "parameter count (Tab. A.1)"}


def paper_main(args, name="paper"):
    """The paper's model and its whole forward as deployed (Sec. 3.1-3.3, 4.2): per
    step the fp64 seed writes its three features into the 15-feature hit rows in
    place, the encoder (the paper's concatenation topology with endpoint readout,
    or the Transformer of its encoder comparison, fp16 operands) runs, and the
    decode turns the median corrections into track parameters.  The paper's
    figures (H100 NVL, its own kernels and data) are context, not a baseline for
    this workload."""
    import torch
    from paper_2609_32479_gb300 import trackfit as TF
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = W.workload(name, n_tracks=args.n_tracks)
    m = w.model
    tb = W.gen_tracks(w)
    blob = W.gen_weights(m, w.weight_seed)
    B = w.n_tracks
    hits = torch.from_numpy(W.paper_hits(tb, w)).to(dev)
    nh = torch.from_numpy(tb.n_hits).to(dev)
    seed = torch.empty((B, 5), dtype=torch.float64, device=dev)
    corr = torch.empty((B, 5), dtype=torch.float32, device=dev)
    out = torch.empty((B, 5), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    reps = max(args.steps, 3)
    with TF.Trackfit(m, blob) as tf:
        def step():
            TF.seed(hits, nh, w.b_field, seed, stream=stream, in_place_at=12)
            tf.forward(hits, nh, corr, stream)
            TF.decode(seed, corr, out, stream)
        for _ in range(max(args.warmup, 1)):
            step()
        ms = _time_events(step, reps, stream)
        enc_ms = _time_events(lambda: tf.forward(hits, nh, corr, stream), reps, stream)
        # the product kernel's own launches, timed by the library's hook in a
        # separate pass (the hook synchronises between batches of launches)
        tf.profile(True)
        tf.profile_read()
        for _ in range(reps):
            tf.forward(hits, nh, corr, stream)
        kern_ms, kern_n = tf.profile_read()
        tf.profile(False)
        st, nbad = tf.device_errors(stream)
        path = tf.path
    D, H = m.d_model, m.d_hidden
    if path.startswith("tcgen05-rows"):
        # the products are contractions of K = 128-480 with fp32 results: far below
        # the tensor pipe's ridge point, so HBM bounds them
        peaks, peak_kind = load_peaks()
        peak = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
        ach = reps * product_bytes(m, tb.n_hits) / (kern_ms * 1e-3) / 1e9
        tfl = reps * product_flops(m, tb.n_hits) / (kern_ms * 1e-3) / 1e12
        roof = {"bound": "hbm", "kernel": "row_gemm_kernel (tcgen05 fp16 products over valid hit rows)",
                "achieved": ach, "peak": peak, "unit": "GB/s", "frac": ach / peak, "traffic": None,
                "peak_kind": f"{peak_kind} copy bandwidth",
                "bytes_per_valid_hit": product_bytes(m, [1]), "tensor_tflops": tfl,
                "launches_per_step": kern_n // reps, "kernel_ms_per_step": kern_ms / reps}
    else:
        ach = encoder_flops(m, tb.n_hits) / (enc_ms * 1e-3) / 1e12
        roof = {"bound": "alu", "kernel": "CUDA-core encoder (fp32 FMA, 16-bit operands)", "achieved": ach,
                "peak": FP32_ALU_TFLOPS, "unit": "TFLOP/s", "frac": ach / FP32_ALU_TFLOPS,
                "peak_kind": "derived: 152 SMs x 128 FP32 lanes x 2 x 2.07 GHz"}
    topo = {W.TOPOLOGY_CONCAT: "concat", W.TOPOLOGY_ATTENTION: "attention"}.get(m.topology, "merge")
    what = "the paper's model" if name == "paper" else "the paper's Transformer encoder"
    line = {"metric": f"tracks/sec at 1 GB300, {what} and seed-guided forward (device-timed)",
            "value": B / (ms * 1e-3), "unit": "tracks/s", "n_gpus": 1, "steps": reps, "warmup": max(args.warmup, 1),
            "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f16",
            "data": "synthetic helix tracks + random-init weights (seeded)", "path": path,
            "config": {"workload": name, "n_tracks": B, "max_hits": m.max_hits, "n_features": m.n_features,
                       "d_model": D, "d_hidden": H, "n_layers": m.n_layers, "topology": topo,
                       "pool": "endpoints" if m.pool == W.POOL_ENDPOINTS else "mean",
                       "l2": "inputs larger than L2; no flush", "parameters": W.weight_count(m)},
            "encoder_ms": enc_ms, "seed_and_decode_ms": ms - enc_ms,
            "roofline": roof,
            "context": PAPER_CONTEXT[name],
            "device_errors": {"status": st, "bad_tracks": nbad}}
    print(json.dumps(line))
    return 0


def code_digest(path: str) -> str:
    """sha256 of a CUDA source's code: comments removed and whitespace collapsed, so
    that an edit of the comments alone keeps the digest (the compiled kernel is the
    same) and any change of the code changes it."""
    import re
    with open(path) as fh:
        src = fh.read()
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    src = re.sub(r"//[^\n]*", " ", src)
    return hashlib.sha256(" ".join(src.split()).encode()).hexdigest()


def traffic_for_kernel():
    """dram bytes per launch from the committed ncu summary, if it was taken on the
    current kernel code (else null)."""
    try:
        with open(TRAFFIC_FILE) as fh:
            d = json.load(fh)
        if d.get("kernel_code_sha256") != code_digest(KERNEL_SRC):
            return None
        return float(d["dram_bytes_per_launch_full"])
    except (OSError, KeyError, ValueError):
        return None


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="large")
    ap.add_argument("--n-tracks", type=int, default=None)
    ap.add_argument("--precision", choices=["config", "bf16", "fp16"], default="config")
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true", help="length x batch sweep, one line per point")
    ap.add_argument("--seed", action="store_true", help="time the analytic seed, features and decode")
    ap.add_argument("--packed", action="store_true", help="time the packed-input entry point")
    ap.add_argument("--paper", action="store_true", help="the paper's model, seed-guided forward")
    ap.add_argument("--transformer", action="store_true", help="the paper's Transformer encoder, seed-guided")
    args = ap.parse_args()
    if args.sweep:
        return sweep_main(args)
    if args.paper:
        return paper_main(args)
    if args.transformer:
        return paper_main(args, "transformer")
    kw = {}
    if args.precision != "config":
        kw["precision"] = W.PRECISION_BF16 if args.precision == "bf16" else W.PRECISION_FP16
    w = W.workload(args.workload, n_tracks=args.n_tracks, **kw)
    if args.impl == "reference":
        return reference_main(args, w)
    if args.seed or args.packed:
        return next_main(args, w)

    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    from paper_2609_32479_gb300 import trackfit as TF

    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    m = w.model
    B = w.n_tracks
    tf = TF.Trackfit(m, blob)
    hits = torch.from_numpy(tb.hits).to(dev)
    n_hits = torch.from_numpy(tb.n_hits).to(dev)
    out = torch.empty((B, 5), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    for _ in range(max(args.warmup, 0)):
        tf.forward(hits, n_hits, out, stream)
    torch.cuda.synchronize(dev)
    st, nbad = tf.device_errors(stream)
    if st not in (TF.OK, TF.ERR_BAD_HITS):
        raise RuntimeError(f"device error status {st} during warm-up")

    tf.profile(True)
    tf.profile_read()
    clocks = ClockSampler() if rank == 0 else None
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize(dev)
    if clocks:
        clocks.start()
        time.sleep(0.3)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    ev[0].record(stream)
    for k in range(args.steps):
        tf.forward(hits, n_hits, out, stream)
        ev[k + 1].record(stream)
    torch.cuda.synchronize(dev)
    if dist is not None:
        dist.barrier()
    clk = clocks.stop() if clocks else None
    step_ms = [ev[k].elapsed_time(ev[k + 1]) for k in range(args.steps)]
    total_ms = ev[0].elapsed_time(ev[args.steps])
    kern_ms, kern_n = tf.profile_read()
    tf.profile(False)
    st, nbad = tf.device_errors(stream)
    if dist is not None:
        t = torch.tensor([total_ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    n_ranks = world
    value = n_ranks * B * args.steps / (total_ms * 1e-3)

    # ---- end to end through the C-ABI with host buffers (pinned), copies inside
    gpu_out = out.cpu().numpy()
    e2e_value, same = None, None
    if args.e2e_steps > 0:
        hits_h = torch.from_numpy(tb.hits).pin_memory()
        n_h = torch.from_numpy(tb.n_hits).pin_memory()
        out_h = torch.empty((B, 5), dtype=torch.float32).pin_memory()
        tf.forward_host_ptr(hits_h.data_ptr(), n_h.data_ptr(), B, out_h.data_ptr(), stream)
        if dist is not None:
            dist.barrier()
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            tf.forward_host_ptr(hits_h.data_ptr(), n_h.data_ptr(), B, out_h.data_ptr(), stream)
        e2e_s = time.perf_counter() - t0
        if dist is not None:
            t = torch.tensor([e2e_s], device=dev)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            e2e_s = float(t.item())
        e2e_value = n_ranks * B * args.e2e_steps / e2e_s
        same = bool(np.array_equal(out_h.numpy(), gpu_out))

    if rank != 0:
        tf.close()
        if dist is not None:
            dist.destroy_process_group()
        return 0

    peaks, peak_kind = load_peaks()
    valid_hits = int(tb.n_hits.clip(0, m.max_hits).sum())
    flops = valid_hits * flops_per_hit(m) + B * flops_per_track_head(m)
    kern_avg_s = (kern_ms / max(kern_n, 1)) * 1e-3
    # the library splits a step into launches (1,048,576 tracks each when, as
    # here, no pooled output buffer is passed): per-launch work is the step's share
    launches_per_step = max(kern_n // max(args.steps, 1), 1) if kern_n else 1
    flops_launch = flops / launches_per_step
    dtype_tf = {1: "bf16_tflops", 2: "bf16_tflops"}.get(m.precision, "bf16_tflops")
    peak = float(peaks.get(dtype_tf, FALLBACK_PEAKS["bf16_tflops"]))
    peak_sus = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    achieved = flops_launch / kern_avg_s / 1e12 if kern_n else None
    bound, peak_kind = "tensor", f"{peak_kind} bf16 dense burst (fp16 runs at the bf16 rate)"
    if m.precision == 0:
        # fp32 configs run on the CUDA cores: the denominator is the FP32 FFMA
        # rate derived from unit counts and clock (SMs x 128 lanes x 2 flop x
        # maximum SM clock), not a tensor-core peak
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        mhz = float(peaks.get("sm_max_mhz", 2070.0))
        peak = sms * 128 * 2 * mhz * 1e6 / 1e12
        peak_sus = peak
        bound = "alu"
        peak_kind = f"FP32 FFMA peak derived: {sms} SMs x 128 lanes x 2 flop x {mhz:.0f} MHz"
    # the committed capture is of the fused kernel on the large workload's model
    traffic = traffic_for_kernel() if (tf.path.startswith("tcgen05") and w.name == "large") else None
    if traffic is not None:   # the summary scales its capture to 1,048,576 tracks
        traffic *= (B / launches_per_step) / 1048576
    roofline = {"bound": bound, "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": (achieved / peak) if achieved else None, "traffic": traffic,
                "peak_kind": peak_kind,
                "frac_of_sustained": (achieved / peak_sus) if achieved else None,
                "kernel": "tc_forward_kernel" if tf.path.startswith("tcgen05") else "simt layer sequence",
                "kernel_ms_avg": kern_avg_s * 1e3, "launches_per_step": launches_per_step,
                "flops_per_launch": flops_launch,
                "algorithmic_bytes_per_launch": B * bytes_per_track(m) / launches_per_step,
                "hbm_frac_of_time": (B * bytes_per_track(m) / launches_per_step /
                                     (peaks.get("hbm_gbs", 6800.0) * 1e9)) / kern_avg_s if kern_n else None}
    line = {"metric": METRIC, "value": value, "unit": "tracks/s", "n_gpus": n_ranks, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps,
            "ms_per_step_min": float(min(step_ms)), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": {0: "f32", 1: "bf16", 2: "f16"}[m.precision],
            "data": "synthetic helix tracks + random-init weights (seeded)", "config": config_block(w, tb),
            "path": tf.path, "roofline": roofline, "clocks": clk,
            "e2e": {"value": e2e_value, "unit": "tracks/s", "h2d_bytes_per_step": int(tb.hits.nbytes + tb.n_hits.nbytes),
                    "d2h_bytes_per_step": int(B * 5 * 4), "matches_device_result": same},
            # per launch chunk: three packing kernels, the fused encoder, the head
            "gpu_launches": int(5 * math.ceil(B / 1048576) * args.steps) if tf.path.startswith("tcgen05") else None,
            "device_errors": {"status": st, "bad_tracks": nbad}}
    if not args.no_cpu_baseline and world == 1:
        pool = OraclePool(w)
        v, idx, ref, dt = run_oracle_sample(w, blob, tb, args.cpu_budget, pool)
        pool.close()
        line["cpu_baseline"] = {"value": v, "unit": "tracks/s", "cores": pool.workers, "kind": "oracle",
                                "sample": f"{idx.size} stratified tracks of {w.name} (numpy fp64, {dt:.1f} s; "
                                          f"one single-threaded oracle process per core)"}
        line["parity_on_sample"] = parity_block(w, blob, tb, gpu_out, idx, ref)
    tf.close()
    print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
