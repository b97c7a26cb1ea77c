"""The replica path of the benchmark on CPU: two gloo ranks (world size 2)
run the same barrier / max / sum bookkeeping the GPU ranks use; the
reference arm prints only on rank 0."""
import json
import os
import socket
import subprocess
import sys

import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench

    d = bench.Dist(backend="gloo")
    d.barrier()
    slowest = d.max(10.0 + rank)            # ms of this rank
    gbs = bench.job_gbs(1e9 * (rank + 1), slowest, d)
    d.barrier()
    q.put((rank, slowest, gbs))
    d.close()


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # both ranks agree: slowest rank 11 ms, 3 GB in total -> 3 GB / 11 ms
    for rank, slowest, gbs in out:
        assert slowest == 11.0
        assert abs(gbs - 3.0 / 0.011) < 1e-6


def test_reference_arm_prints_on_rank0_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], capture_output=True, text=True, env=env, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_single_process_dist_is_a_no_op():
    sys.path.insert(0, ROOT)
    import bench

    d = bench.Dist()
    assert not d.on and d.max(3.5) == 3.5 and d.sum(2.0) == 2.0
    assert abs(bench.job_gbs(2e9, 1000.0, d) - 2.0) < 1e-12
    line = {"impl": "reference"}
    assert json.loads(json.dumps(line)) == line


def test_reference_arm_line_has_the_contract_keys():
    """The reference arm (the oracle on the host cores) prints one JSON line
    with the keys of the bench contract."""
    env = {k: v for k, v in os.environ.items() if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK")}
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], capture_output=True, text=True, env=env, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["unit"] == "GB/s" and d["value"] > 0 and d["higher_is_better"] is True
    assert {"value", "unit", "cores", "kind", "sample"} <= set(d["cpu_baseline"])
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert "workload" in d["config"]


def test_host_row_plans_the_oracle_compaction(lib):
    """bench.py's rows.host (the host steps through the control core, no
    GPU): every figure is present and positive, and its compaction plan of
    the 64 GiB fragmentation trace moves exactly the oracle's pages."""
    import bench
    import workloads as W
    from oracle import OracleStore, PutItem

    h = bench.time_host_control(reps=5)
    for k in ("handoff_put_us", "handoff_free_us", "handoff_get_us", "adapter_set_put_us", "adapter_get_256_us",
              "compaction_plan_ms"):
        assert h[k] > 0, k
    assert h["adapter_set_put_evictions_per_call"] > 0
    C5 = W.COMPACTION
    P = C5["page_bytes"]
    tr = W.compaction_trace(1, C5["pool_bytes"] // P, P, C5["n_ops"], C5["lo"], C5["hi"], C5["p_free"],
                            C5["settle_frac"])
    ora = OracleStore(C5["pool_bytes"], P, keep_bytes=False)
    ids = {}
    for op in tr.ops:
        if op[0] == "alloc":
            ids[op[1]] = ora.put_batch([PutItem(op[2])])[1][0]
        else:
            ora.free([ids.pop(op[1])])
    st, moves = ora.compact(C5["limit_bytes"])
    assert st == 0 and h["compaction_moves"] == len(moves)
