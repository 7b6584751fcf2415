"""Multi-rank host logic of bench.py on CPU with the gloo backend (world size 2).

The layer shards by tokens with no data-path exchange: each rank draws its own
batch (seed + rank), the job time is the slowest rank's (a max-reduce, the only
collective besides the barrier), and throughput counts every rank's tokens.
"""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import synth


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = synth.Workload("mr", S=16, GBS=2, D=64, E=4, K=2, F=64)
        x = synth.make_inputs(w, seed=bench.rank_seed(w, rank))["x"]
        xs = [torch.empty_like(x) for _ in range(world)]
        dist.all_gather(xs, x)                        # test-only: compare the ranks' batches
        distinct = not torch.equal(xs[0], xs[1])
        t = bench.max_over_ranks(1.0 + rank, world, "cpu")
        dist.barrier()
        q.put((rank, distinct, t, bench.job_throughput(world, w.T, t)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_tokens_and_take_the_slowest_time():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(world))
    for rank, distinct, t, thr in res:
        assert distinct                              # each rank holds its own tokens
        assert t == 2.0                              # the slowest rank's time on every rank
        assert thr == pytest.approx(world * 32 / 2e-3)


def test_reference_arm_runs_only_on_rank_zero(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setattr(bench, "OracleRunner", lambda *a, **k: pytest.fail("rank 1 must not run the oracle"))

    class A:
        steps, warmup, ref_tokens, gpus = 3, 3, 0, 2
    bench.run_reference(A(), synth.TINY)
    assert capsys.readouterr().out == ""


def test_job_throughput_is_weak_scaling():
    assert bench.job_throughput(4, 8192, 2.0) == pytest.approx(4 * bench.job_throughput(1, 8192, 2.0))


def test_step_statistics_filters_outliers_iteratively():
    """The filtered mean removes steps above mean + 1.5 sd until none is left:
    one slow step (10) is removed first; the next pass then removes the
    moderate one (2) that the first pass's wide sd let through."""
    steps = [1.0] * 20 + [2.0, 10.0]
    st = bench.step_statistics(steps)
    assert st["dropped"] == 2
    assert st["filtered_mean_ms"] == 1.0
    assert st["median_ms"] == 1.0 and st["max_ms"] == 10.0
    assert bench.step_statistics([1.0, 1.0, 1.0])["dropped"] == 0


def test_every_timed_kernel_has_algorithmic_work():
    """Each kernel the library times (KernelScope names and the tensor-core
    GEMM names in the C sources) has a roofline entry in bench.kernel_work,
    except the few that do no algorithmic work of the method."""
    import glob
    import re
    import synth
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    names = set()
    for f in glob.glob(os.path.join(root, "paper_2608_28511_gb300", "csrc", "*.cu")):
        text = open(f).read()
        names |= set(re.findall(r'KernelScope ks\("([a-z0-9_]+)"', text))
        names |= set(re.findall(r'"([a-z0-9_]+_tc)"', text))
    no_work = {"group_maps", "sum_splits", "pack_w1", "perm_zero", "balance_finalize"}
    w = synth.get("C4")
    missing = [n for n in sorted(names - no_work) if bench.kernel_work(n, w, w.T, 2688)[1] <= 0]
    assert not missing, missing
    assert len(names) >= 30


_TINY_CU = 'extern "C" __global__ void tiny_kernel(int* p) { p[threadIdx.x] = 1; }\n' \
           'extern "C" int tiny_version(void) { return 7; }\n'


def _build_worker(rank, world, port, root, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import functools
        from paper_2608_28511_gb300 import _build
        fn = functools.partial(_build.build, csrc=os.path.join(root, "csrc"), build_dir=os.path.join(root, "obj"),
                               lib=os.path.join(root, "libtiny.so"))
        bench.gated_build(world, rank, dist.barrier, build_fn=fn)
        dist.barrier()
        q.put((rank, [os.path.basename(s) for s in _build.last_compiled]))
    finally:
        dist.destroy_process_group()


def test_gated_build_compiles_stale_objects_once_per_node(tmp_path):
    """Two ranks start a build over an object older than its source: local rank
    0 recompiles and links while rank 1 waits, then rank 1 finds everything up
    to date.  No temporary file is left behind."""
    import shutil
    import time
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_2608_28511_gb300 import _build
    root = str(tmp_path)
    os.makedirs(os.path.join(root, "csrc"))
    src = os.path.join(root, "csrc", "tiny.cu")
    with open(src, "w") as f:
        f.write(_TINY_CU)
    lib = os.path.join(root, "libtiny.so")
    _build.build(csrc=os.path.join(root, "csrc"), build_dir=os.path.join(root, "obj"), lib=lib)
    time.sleep(1.1)
    os.utime(src)                                  # the object is now stale
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_build_worker, args=(r, world, port, root, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
        assert p.exitcode == 0
    res = dict(q.get(timeout=10) for _ in range(world))
    assert res[0] == ["tiny.cu"]                  # rank 0 rebuilt the stale unit
    assert res[1] == []                            # rank 1 found it fresh
    assert os.path.getmtime(os.path.join(root, "obj", "tiny.o")) >= os.path.getmtime(src)
    assert not [n for n in os.listdir(root) + os.listdir(os.path.join(root, "obj")) if n.endswith(".tmp")]
