"""The N > 1 path on CPU: two gloo ranks run independent replicas.

Token rows are independent on the whole hot path, so N GPUs run N replicas
with no data-path collective (replicas.py); these tests run the host-side
parts of that path with world_size 2 on the gloo backend: per-rank inputs,
a replica of the rotate+quant -> GEMM chain on each rank (the oracle stands
in for the device kernels, which need a GPU), the max-over-ranks timing and
the whole-job rate.
"""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

from paper_2405_16406_gb300 import replicas, synth


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _replica(rank: int, world: int, port: int, out_dir: str) -> None:
    import torch
    import torch.distributed as dist

    import oracle

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each rank draws its own tokens; the weights are the same everywhere
        rng = np.random.default_rng(replicas.input_seed(100, rank))
        x = synth.activations(rng, 8, 256, outlier_count=4, factor=50.0)
        w = synth.weights(np.random.default_rng(7), 64, 256)
        qa = oracle.rotate_quant_act(x, (1, 256), 4, True, 1.0)
        qw = oracle.quant_weight(w, (1, 256))
        y = oracle.w4a4_linear(qa, qw).y
        replicas.barrier(world)
        # the slowest rank sets the job's time
        t_local = 0.010 * (rank + 1)
        t_max = replicas.max_over_ranks(t_local, world)
        rate = replicas.whole_job_rate(8, t_max, world)
        np.savez(os.path.join(out_dir, f"rank{rank}.npz"), x=x, y=y, t_max=t_max, rate=rate)
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_gloo_replicas(tmp_path):
    world, port = 2, _free_port()
    mp.start_processes(_replica, args=(world, port, str(tmp_path)), nprocs=world, start_method="spawn", join=True)
    import oracle
    res = [np.load(tmp_path / f"rank{r}.npz") for r in range(world)]
    # distinct inputs per rank
    assert not np.array_equal(res[0]["x"], res[1]["x"])
    w = synth.weights(np.random.default_rng(7), 64, 256)
    qw = oracle.quant_weight(w, (1, 256))
    for r in range(world):
        # each rank's result is exactly what one process computes for its tokens
        rng = np.random.default_rng(replicas.input_seed(100, r))
        x = synth.activations(rng, 8, 256, outlier_count=4, factor=50.0)
        assert np.array_equal(res[r]["x"], x)
        y = oracle.w4a4_linear(oracle.rotate_quant_act(x, (1, 256), 4, True, 1.0), qw).y
        assert np.array_equal(res[r]["y"], y)
        # both ranks agree on the maximum time and the whole-job rate
        assert float(res[r]["t_max"]) == pytest.approx(0.020)
        assert float(res[r]["rate"]) == pytest.approx(2 * 8 / 0.020)


def test_single_rank_needs_no_process_group():
    assert replicas.max_over_ranks(3.5, 1) == 3.5
    replicas.barrier(1)
    assert replicas.whole_job_rate(10, 2.0, 1) == 5.0
    with pytest.raises(ValueError):
        replicas.whole_job_rate(10, 0.0, 2)
