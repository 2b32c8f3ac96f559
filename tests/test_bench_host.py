"""Host-side logic of bench.py on CPU: the replica timing reduction over a
world-size-2 gloo group, the clock-sample parsing, and the reference arm's
JSON line (the CPU oracle timed on a bounded sample)."""
import json
import os
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      ORDERMOE_BENCH_BACKEND="gloo")
    sys.path.insert(0, ROOT)
    import bench
    d = bench.Dist()
    d.barrier()
    m = d.max(10.0 + rank)
    q.put((rank, m))
    d.close()


def test_replica_timing_takes_the_max_over_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29000 + os.getpid() % 1000
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(60)
        assert p.exitcode == 0
    assert res == {0: 11.0, 1: 11.0}


def test_clock_sample_parsing(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench

    class FakeProc:
        def terminate(self):
            pass

        def communicate(self, timeout=None):
            rows = ["0, 1900, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
                    "0, 1950, 2070, 1000.0, 0x4, Not Active, Not Active, Not Active, Active",
                    "0, 1800, 2070, 1100.0, 0x4, Not Active, Not Active, Not Active, Active"]
            return "\n".join(rows), ""

    s = bench.ClockSampler("0")
    s.proc = FakeProc()
    c = s.stop()
    assert c == {"sm_mhz": 1900.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}


def test_reference_arm_prints_the_contract_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--workload", "tiny", "--steps", "2", "--warmup", "1"],
                       capture_output=True, text=True, env=env, timeout=600)
    assert r.returncode == 0, r.stderr
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "tokens/s" and line["value"] > 0
    assert line["higher_is_better"] is True
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1


def test_tensor_peak_follows_the_run():
    """The bf16 peak a tensor-bound fraction divides by: the burst figure for
    a short region with no power cap seen, the sustained one otherwise; both
    fractions are printed and the one that applies is named."""
    sys.path.insert(0, ROOT)
    import bench
    pk = {"bf16_tflops": 1918.0, "bf16_tflops_sustained": 1723.6}
    quiet = {"reasons": []}
    capped = {"reasons": ["sw_power_cap"]}
    assert bench.tensor_peak(pk, "measured", quiet, 0.036)[:2] == (1918.0, "burst")
    assert bench.tensor_peak(pk, "measured", capped, 0.036)[:2] == (1723.6, "sustained")
    assert bench.tensor_peak(pk, "measured", quiet, 2.0)[:2] == (1723.6, "sustained")
    r = bench.tensor_roofline("k", 1700.0, pk, "measured", quiet, 0.036, traffic=None)
    assert r["peak_applies"] == "burst" and r["frac"] == round(1700.0 / 1918.0, 4)
    assert r["frac_burst"] == round(1700.0 / 1918.0, 4)
    assert r["frac_sustained"] == round(1700.0 / 1723.6, 4)
    assert r["peak_source"] == "measured bf16_tflops" and r["traffic"] is None
