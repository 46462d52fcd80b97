"""The multi-process path of the benchmark on the host: world size 2 over gloo.  Each rank loads
its own replica (nothing in the path is exchanged); the collectives only serve the timing, so
what is checked is the barrier, the maximum of the ranks' times, the sum of their bytes, the
whole-job figure built from them, and that under torchrun only rank 0 prints the reference
arm's line."""
import json
import multiprocessing as mp
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                       "WORLD_SIZE": str(world), "RANK": str(rank), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import bench
    r = bench.Ranks("gloo", "cpu")
    r.barrier()
    got = {"rank": r.rank, "world": r.world,
           "max": r.max(10.0 * (rank + 1)),
           "sum": r.sum(1e9 * (rank + 1)),
           # rank k moved (k + 1) GB in (k + 1) * 100 ms: 3 GB over the slowest 200 ms
           "gbs": bench.whole_job_gbs(r, 1e9 * (rank + 1), 100.0 * (rank + 1))}
    r.barrier()
    r.close()
    out.put(got)


def test_rank_collectives_over_gloo():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(k, 2, port, out)) for k in range(2)]
    for p in procs:
        p.start()
    res = [out.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert sorted(x["rank"] for x in res) == [0, 1]
    for x in res:
        assert x["world"] == 2
        assert x["max"] == 20.0
        assert x["sum"] == 3e9
        assert abs(x["gbs"] - 15.0) < 1e-9


def test_single_process_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    saved = {k: os.environ.pop(k, None) for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK")}
    try:
        r = bench.Ranks("gloo", "cpu")
        assert (r.world, r.rank) == (1, 0)
        assert r.max(3.5) == 3.5 and r.sum(7) == 7.0
        assert abs(bench.whole_job_gbs(r, 2e9, 500.0) - 4.0) < 1e-12
        r.barrier()
        r.close()
    finally:
        for k, v in saved.items():
            if v is not None:
                os.environ[k] = v


@pytest.mark.slow
def test_reference_arm_under_torchrun_prints_one_line():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "2", "--warmup", "1",
           "--workload", "tiny_1000"]
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [json.loads(x) for x in p.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["steps"] == 2
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"


def test_bench_labels_and_traffic_record(monkeypatch):
    """The benchmark's dtype label and dominant work class come from the workload; the recorded
    ncu traffic is reported only while the kernel sources match the capture."""
    sys.path.insert(0, ROOT)
    import bench
    import workloads
    assert bench.path_types(workloads.named_config("llama3_8b_bf16"))[:2] == ("u16", 1)
    assert bench.path_types(workloads.named_config("llama3_8b_f32_rne"))[:2] == ("f32->bf16", 4)
    dt, cls, _ = bench.path_types(workloads.named_config("llama3_8b_fp8_block128"))
    assert dt == "u16+u32+u8" and cls == 0
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        name, rec = next(iter(json.load(f).items()))
    monkeypatch.setattr(bench, "kernel_source_hash", lambda files=None: rec["kernel_sha256"])
    assert bench.recorded_traffic(name) == rec["dram_bytes_per_launch"]
    monkeypatch.setattr(bench, "kernel_source_hash", lambda files=None: "0" * 64)
    assert bench.recorded_traffic(name) is None
    assert bench.recorded_traffic("no_such_workload") is None
    # a record names the sources of the kernel it captured; the hash covers those only
    monkeypatch.undo()
    files = tuple(rec.get("sources", bench.KERNEL_SOURCES))
    assert len(bench.kernel_source_hash(files)) == 64
    st = {"n_bulk": 3, "n_slabs": 0, "n_tiny": 5, "n_strided": 0}
    assert bench.kernel_names(st) == "cfa_bulk_kernel (TMA bulk copies) + cfa_tiny_kernel (tiny pieces)"


def test_attribution_sizes_fit_any_checkpoint():
    """The pageable H2D and host memcpy measurements never slice past a checkpoint smaller than
    their 1 and 4 GiB buffers, and split the memcpy evenly among the threads."""
    import bench
    gib = 1 << 30
    for size, threads in [(16_060_000_000, 16), (16_060_000_000, 12), (1_396_744_192, 16),
                          (125 << 20, 72), (100, 16), (7, 16), (0, 4)]:
        n_h2d, part = bench.attribution_sizes(size, threads)
        assert n_h2d == min(gib, size)
        assert part * threads <= min(4 * gib, size)
        assert min(4 * gib, size) - part * threads < threads
