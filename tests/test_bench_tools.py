"""Host-side tools of bench.py (no GPU): recording ncu's DRAM traffic for the
current kernel source and finding it again."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

HEADER = ('"ID","Process ID","Process Name","Host Name","Kernel Name","Context","Stream","Block Size",'
          '"Grid Size","Device","CC","Section Name","Metric Name","Metric Unit","Metric Value"')


def _row(i, kernel, metric, unit, value):
    return (f'"{i}","1","python3","h","{kernel}","1","7","(128, 1, 1)","(4096, 1, 1)","0","10.3",'
            f'"Command line profiler metrics","{metric}","{unit}","{value}"')


def test_record_traffic_from_an_ncu_csv(tmp_path, monkeypatch):
    import bench
    k = "void <unnamed>::sc_unit_kernel<unsigned short, false>(<unnamed>::Params)"
    lines = ["==PROF== Connected to process 1", HEADER,
             _row(0, "void at::native::FillFunctor<unsigned char>", "dram__bytes_read.sum", "byte", "7"),
             _row(1, k, "dram__bytes_read.sum", "Mbyte", "1,079.37"),
             _row(1, k, "dram__bytes_write.sum", "Kbyte", "3,649.28"),
             _row(1, k, "gpu__time_duration.sum", "usecond", "195.5"),
             _row(2, k, "dram__bytes_read.sum", "byte", "5")]
    csv_path = tmp_path / "traffic.csv"
    csv_path.write_text("\n".join(lines) + "\n")
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(tmp_path / "traffic.json"))
    e = bench.record_traffic(str(csv_path), "cfgX: a workload", "ncu ... python bench.py")
    assert e["dram_bytes_read"] == 1_079_370_000 and e["dram_bytes_write"] == 3_649_280
    assert e["dram_bytes_per_launch"] == 1_079_370_000 + 3_649_280
    assert e["kernel_sha"] == bench.kernel_sha()
    assert bench.stored_traffic("cfgX: a workload") == e["dram_bytes_per_launch"]
    assert bench.stored_traffic("another workload") is None
    # an entry recorded for other kernel code is not used
    d = json.loads((tmp_path / "traffic.json").read_text())
    d["cfgX: a workload"]["kernel_sha"] = "0" * 16
    (tmp_path / "traffic.json").write_text(json.dumps(d))
    assert bench.stored_traffic("cfgX: a workload") is None


def test_step_spread_matches_linear_percentiles():
    import numpy as np

    import bench
    rng = np.random.default_rng(5)
    for n in (1, 2, 7, 50):
        xs = list(rng.uniform(0.1, 0.3, n))
        s = bench.step_spread(xs)
        assert s["n"] == n
        for key, q in (("p10", 10), ("median", 50), ("p90", 90)):
            assert abs(s[key] - float(np.percentile(xs, q))) < 1e-12
    assert bench.step_spread([])["median"] is None


def _bench_lines(args, env=None):
    import subprocess
    e = dict(os.environ)
    e.update(env or {})
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], capture_output=True,
                         text=True, timeout=600, cwd=ROOT, env=e)
    assert out.returncode == 0, out.stderr[-2000:]
    return [json.loads(ln) for ln in out.stdout.splitlines() if ln.startswith("{")]


def test_reference_arm_prints_the_contract_line():
    # the reference arm (the oracle on the host cores) on the smallest named
    # workload: one JSON line with the bench's metric, the oracle as the CPU
    # baseline and an end-to-end figure that moves no bytes to or from a GPU
    lines = _bench_lines(["--impl", "reference", "--config", "1", "--steps", "2", "--warmup", "3"])
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference" and d["metric"] == "verified positions/s"
    assert d["unit"] == "positions/s" and d["higher_is_better"] is True
    assert d["steps"] == 2 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["vs_baseline"] is None
    assert d["config"]["B"] == 8 and d["config"]["gamma"] == 5 and d["config"]["V"] == 32128
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "positions/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_reference_arm_prints_on_rank_zero_only():
    # under torchrun only rank 0 runs the oracle and prints; the other ranks exit 0
    assert _bench_lines(["--impl", "reference", "--config", "1", "--steps", "1", "--warmup", "3"],
                        {"RANK": "1", "LOCAL_RANK": "1", "WORLD_SIZE": "2"}) == []
