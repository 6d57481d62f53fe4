"""bench.py's reference arm (the CPU oracle, timed on the host cores) keeps the JSON
contract the driver reads; it runs without a GPU."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_line_on_the_tiny_workload():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--workload", "tiny_f32_nchw", "--steps", "2", "--warmup", "1"],
                         capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "config", "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["value"] > 0 and line["steps"] == 2 and line["warmup"] == 1
    assert line["config"]["workload"] == "tiny_f32_nchw"
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["e2e"]["value"] == line["value"]


def test_oracle_on_every_core_covers_the_sample():
    import importlib.util

    from paper_2608_23794_gb300 import synth
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    bench = importlib.util.module_from_spec(spec)
    sys.modules["bench"] = bench
    spec.loader.exec_module(bench)
    import oracle
    oracle.build()
    cfg = synth.CONFIGS["rn50_stage1_reduce"].replace(N=5, H=6, W=6)
    pool = bench.OraclePool(cfg, 0, 5, 4)
    try:
        # the jobs cover examples 0..4 once, rows [0, 4)
        assert sorted(j[:2] for j in pool.jobs)[0][0] == 0
        assert sum(e1 - e0 for e0, e1, _ in pool.jobs) == 5
        assert all(h == 4 for _, _, h in pool.jobs)
        assert sum(pool.pool.map(bench._pool_run, pool.jobs)) == 5
        assert pool.run() > 0
    finally:
        pool.close()
    t, procs = bench.oracle_parallel_run(cfg, 0, 5, 6, 0.2)
    assert t > 0 and 1 <= procs <= 5
