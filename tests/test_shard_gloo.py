"""Replica sharding across ranks (gloo, world size 2, CPU): every rank computes its
contiguous slice of the batch and the gathered result equals one un-sharded run."""
import dataclasses
import os

import numpy as np
import pytest
import torch.multiprocessing as mp

from paper_2609_32479_gb300.shard import shard_range


@pytest.mark.parametrize("n,world", [(10, 2), (11, 2), (1, 2), (7, 3), (1000, 4)])
def test_shard_ranges_partition_the_batch(n, world):
    spans = [shard_range(n, r, world) for r in range(world)]
    assert spans[0][0] == 0 and spans[-1][1] == n
    for (b0, e0), (b1, e1) in zip(spans, spans[1:]):
        assert e0 == b1
    sizes = [e - b for b, e in spans]
    assert max(sizes) - min(sizes) <= 1


def _worker(rank, world, port, path):
    import torch.distributed as dist
    from oracle import trackfit_oracle as O
    from paper_2609_32479_gb300 import workloads as W
    from paper_2609_32479_gb300.shard import gather_outputs
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w = W.workload("tiny", n_tracks=37)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, 1)
    b, e = shard_range(37, rank, world)
    local = O.forward(dataclasses.asdict(w.model), blob, tb.hits[b:e], tb.n_hits[b:e])
    full = gather_outputs(local, 37)
    if rank == 0:
        np.save(path, full)
    dist.barrier()
    dist.destroy_process_group()


def test_gloo_two_rank_shard_and_gather(tmp_path):
    import socket
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    path = str(tmp_path / "full.npy")
    mp.start_processes(_worker, args=(2, port, path), nprocs=2, start_method="spawn", join=True)
    from oracle import trackfit_oracle as O
    from paper_2609_32479_gb300 import workloads as W
    w = W.workload("tiny", n_tracks=37)
    tb = W.gen_tracks(w)
    ref = O.forward(dataclasses.asdict(w.model), W.gen_weights(w.model, 1), tb.hits, tb.n_hits)
    np.testing.assert_allclose(np.load(path), ref, rtol=1e-12, atol=1e-14)
