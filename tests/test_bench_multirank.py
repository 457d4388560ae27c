"""The bench's N > 1 logic on CPU: two ranks over gloo (127.0.0.1).

`bench.py --gpus N` runs one process per GPU, each stepping its own full parameter
set (weak scaling, no data-path collective). The job's step time is the slowest
rank's, and the job's throughput counts every rank's parameters; the reference
arm runs on rank 0 only. These are checked here with the bench's own functions.
"""
import importlib.util
import os
import socket

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        b = _bench()
        local_ms = [12.5, 9.75][rank]                 # rank 0 is the slow one
        ms = b.max_over_ranks(local_ms, world, torch.device("cpu"))
        rate = b.job_rate(world, 1_000_000, ms)
        with open(os.path.join(out_dir, f"r{rank}.txt"), "w") as f:
            f.write(f"{ms!r} {rate!r}\n")
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_count_every_rank(tmp_path):
    import torch.multiprocessing as mp
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, str(tmp_path))) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = [tuple(float(x) for x in open(tmp_path / f"r{r}.txt").read().split()) for r in range(world)]
    for ms, rate in got:
        assert ms == 12.5                                   # max over ranks
        assert rate == pytest.approx(2 * 1_000_000 / 12.5e-3)  # both ranks' parameters / job time


def test_one_rank_passes_its_own_time_through():
    b = _bench()
    assert b.max_over_ranks(3.25, 1, None) == 3.25
    assert b.job_rate(1, 500, 2.0) == pytest.approx(250_000.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    b = _bench()
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")

    class Args:
        workload, steps, warmup, seed, gpus, ref_seconds = "toy", 1, 0, 0, 2, 1.0
    b.run_reference(Args())                                 # returns before any work or output
    assert capsys.readouterr().out == ""


@pytest.mark.parametrize("n_groups", [1, 2, 4, 8, 1000])
def test_e2e_groups_partition(n_groups):
    """The end-to-end leg's tensor groups: consecutive runs covering every tensor once,
    at most n_groups of them, of about equal bytes on the App. B shapes."""
    b = _bench()
    from paper_2607_19058_gb300 import workloads as WL
    for wl in (WL.appb(), WL.toy()):
        offs, total = [], 0
        for s in wl.specs:
            total = (total + 511) // 512 * 512
            offs.append(total)
            total += s.numel * (4 if s.fp32 else 2)
        offs.append(total)
        groups = b.e2e_groups(offs, n_groups)
        n = len(wl.specs)
        assert 1 <= len(groups) <= min(n_groups, n)
        assert groups[0][0] == 0 and groups[-1][1] == n
        assert all(k1 == k0n for (_, k1), (k0n, _) in zip(groups, groups[1:]))
        assert all(k0 < k1 for k0, k1 in groups)
        if wl.name == "appb" and n_groups <= 8:
            sizes = [(offs[k1] if k1 < n else offs[-1]) - offs[k0] for k0, k1 in groups]
            assert max(sizes) <= 1.1 * total / len(groups)
