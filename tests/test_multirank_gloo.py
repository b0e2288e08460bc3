"""Multi-rank host logic of the benchmark on CPU: world size 2 over gloo.

The path shards with no collective on the data: rank r generates and solves
instances [r*B, (r+1)*B) of the seeded stream, and the timing is the slowest
rank's. These tests run the benchmark's own helpers (`bench.rank_config`,
`bench.max_over_ranks`) in two processes and check, with the oracle, that the
shards together are exactly the world-size batch solved in one process.
"""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

WORLD = 2
B = 48


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out_dir: str, workload: str):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        import oracle
        from paper_2101_07968_gb300 import workloads as wl

        base = wl.with_batch(wl.config(workload), B)
        cfg = bench.rank_config(base, rank)
        prof = oracle.profile_gen(cfg)
        res = {}
        for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
            out = oracle.schedule_batch(d, prof[c], prof[x], prof["dt"], nthreads=1)
            res[d] = (out["makespan"], out["bits"], out["nseg"])
        gathered = [None] * world
        dist.all_gather_object(gathered, (rank, prof["fc"], prof["dt"], res))
        slowest = bench.max_over_ranks(10.0 + rank)  # rank r "took" 10 + r ms
        if rank == 0:
            np.save(os.path.join(out_dir, "slowest.npy"), np.array([slowest]))
            for r, fc, dtv, rr in gathered:
                np.save(os.path.join(out_dir, f"fc{r}.npy"), fc)
                np.save(os.path.join(out_dir, f"dt{r}.npy"), dtv)
                for d in (0, 1):
                    for j, name in enumerate(("makespan", "bits", "nseg")):
                        np.save(os.path.join(out_dir, f"{name}{r}_{d}.npy"), rr[d][j])
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("workload", ["tiny", "vgg16"])
def test_two_rank_shards_equal_one_process(tmp_path, workload):
    import oracle
    from paper_2101_07968_gb300 import workloads as wl

    oracle.build()
    mp.spawn(_rank_main, args=(WORLD, _free_port(), str(tmp_path), workload), nprocs=WORLD,
             join=True)
    assert float(np.load(tmp_path / "slowest.npy")[0]) == 10.0 + (WORLD - 1)

    full = wl.with_batch(wl.config(workload), WORLD * B)
    prof = oracle.profile_gen(full)
    fc = np.concatenate([np.load(tmp_path / f"fc{r}.npy") for r in range(WORLD)])
    dtv = np.concatenate([np.load(tmp_path / f"dt{r}.npy") for r in range(WORLD)])
    assert np.array_equal(fc, prof["fc"]) and np.array_equal(dtv, prof["dt"])
    for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
        exp = oracle.schedule_batch(d, prof[c], prof[x], prof["dt"], nthreads=2)
        for name in ("makespan", "bits", "nseg"):
            got = np.concatenate([np.load(tmp_path / f"{name}{r}_{d}.npy") for r in range(WORLD)])
            assert np.array_equal(got, exp[name]), (workload, d, name)


def test_rank_config_ranges_are_disjoint_and_cover():
    import bench
    from paper_2101_07968_gb300 import workloads as wl

    base = wl.with_batch(wl.config("resnet50"), 1000)
    spans = [(c["inst0"], c["inst0"] + c["batch"]) for c in
             (bench.rank_config(base, r) for r in range(8))]
    assert spans[0] == (0, 1000)
    assert all(spans[r][1] == spans[r + 1][0] for r in range(7))
    assert bench.max_over_ranks(3.5) == 3.5  # no process group: the value itself
