"""World-size-2 gloo test of the layer-partitioned multi-GPU path (no GPU).

The weight path shards by matrix with no data exchange: each rank owns a block
of global matrix indices and regenerates every Z and Omega from the shared seed
and the global index.  This checks, across two real processes, that the
partitions are disjoint and cover the set, that a rank's random streams equal
those a single process computes for the same global indices, and that bench.py's
timing reduction -- the max over ranks of the timed region and the whole-job
throughput world x K / slowest rank -- works over the process group, with a stub
standing in for the library (each rank reports its own region length)."""

import os

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2608_15665_gb300 import workloads


def _worker(rank, world, port, result_path):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from oracle import rng
    wl = workloads.get("lora_opt13b_f32_r4")
    part = workloads.partition(wl, rank, world)
    idx = torch.tensor(list(part["global_indices"]), dtype=torch.int64)
    gathered = [torch.zeros_like(idx) for _ in range(world)]
    dist.all_gather(gathered, idx)
    # the first matrix of this rank: its step-3 Z for query 1 and its refresh-0 Omega_U rows
    g0 = part["matrix_index_base"]
    z = torch.from_numpy(rng.gen_Z(part["seed"], g0, 3, 1, wl.r))
    om = torch.from_numpy(rng.gen_omega(part["seed"], g0, 0, "U", 8, wl.r))
    zs = [torch.zeros_like(z) for _ in range(world)]
    oms = [torch.zeros_like(om) for _ in range(world)]
    dist.all_gather(zs, z)
    dist.all_gather(oms, om)
    t = torch.tensor([float(rank + 1)], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    # bench.py's reduction: a stub timed region per rank (the slower rank 1 sets the pace)
    import bench
    K, F, refresh_ms = 20, 25, 1.3
    stub_ms = 700.0 + 50.0 * rank
    slowest = bench.max_over_ranks(stub_ms, world, "cpu")
    value = bench.job_steps_per_second(bench.amortise_refresh(slowest, K, 5, F, refresh_ms), world)
    if rank == 0:
        torch.save({"idx": gathered, "z": zs, "om": oms, "max": float(t.item()),
                    "slowest": slowest, "value": value}, result_path)
    dist.barrier()
    dist.destroy_process_group()


def test_partition_over_two_gloo_ranks(tmp_path):
    import socket
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    out = str(tmp_path / "res.pt")
    mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
    res = torch.load(out)
    wl = workloads.get("lora_opt13b_f32_r4")
    allidx = torch.cat(res["idx"]).numpy()
    assert np.array_equal(np.sort(allidx), np.arange(2 * wl.n_mats))
    assert len(set(res["idx"][0].tolist()) & set(res["idx"][1].tolist())) == 0
    from oracle import rng
    for r in range(2):
        g0 = r * wl.n_mats
        assert np.array_equal(res["z"][r].numpy(), rng.gen_Z(wl.seed, g0, 3, 1, wl.r))
        assert np.array_equal(res["om"][r].numpy(), rng.gen_omega(wl.seed, g0, 0, "U", 8, wl.r))
    assert not np.array_equal(res["z"][0].numpy(), res["z"][1].numpy())
    assert res["max"] == 2.0
    assert res["slowest"] == 750.0
    assert res["value"] == pytest.approx(2 * 1e3 / (750.0 / 20 + 1.3 / 25))


def test_partition_rejects_bad_rank():
    wl = workloads.get("single256_f32_r8")
    with pytest.raises(ValueError):
        workloads.partition(wl, 2, 2)
