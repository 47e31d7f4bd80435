"""bench.py's reference arm (the CPU oracle timed on bounded samples) runs without
a GPU and prints one JSON line in the contract's shape."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1", "--warmup", "0",
           "--workload", "medium", "--n-tracks", "4096"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["value"] > 0 and d["unit"] == "tracks/s" and d["higher_is_better"] is True
    assert d["config"]["workload"] == "medium"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": "tracks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_oracle_pool_matches_one_process():
    """The CPU baseline's process pool (the oracle on every core, tracks in chunks)
    returns what one call of the oracle returns on the same tracks, in order: equal
    up to the fp64 rounding that a matrix product's blocking over a different batch
    size changes (1e-13 relative measured; 1e-11 allowed)."""
    import dataclasses
    import numpy as np
    sys.path.insert(0, ROOT)
    import bench
    from oracle import trackfit_oracle as O
    from paper_2609_32479_gb300 import workloads as W
    w = W.workload("small", n_tracks=150)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    ref = O.forward(dataclasses.asdict(w.model), blob, tb.hits, tb.n_hits)
    pool = bench.OraclePool(w)
    try:
        got = pool.forward(tb.hits, tb.n_hits, chunk=32)
    finally:
        pool.close()
    assert pool.workers >= 1
    assert got.shape == ref.shape
    np.testing.assert_allclose(got, ref, rtol=1e-11, atol=1e-13)
