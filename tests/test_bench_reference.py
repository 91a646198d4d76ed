"""bench.py on the CPU.  The reference arm (the float64 oracle on the host cores) keeps the JSON
contract: one line with the metric, unit, direction, config, a cpu_baseline describing the run
and an e2e object with no host-device bytes (run on the 2k-node workload).  The ncu traffic
counters are used only for the sources they were taken on, and the operator's algorithmic bytes
follow their definition."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config",
                          "ring_chords_n2000", "--steps", "2", "--warmup", "1"], cwd=ROOT,
                         capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "edges/s" and d["higher_is_better"] is True
    assert d["steps"] == 2 and d["warmup"] == 1 and d["value"] > 0 and d["ms_per_step"] > 0
    assert d["config"]["workload"] == "ring_chords_n2000" and d["config"]["precond"] == "none"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1
    assert cb["sample"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_traffic_is_reported_only_for_the_captured_sources(tmp_path, monkeypatch):
    """profiles/traffic.json counters are used only while the solver sources hash to the value
    recorded with them; any other hash (a changed kernel) yields null."""
    sys.path.insert(0, ROOT)
    import bench

    sha = bench.solver_src_sha1()
    prof = tmp_path / "profiles"
    prof.mkdir()
    (prof / "traffic.json").write_text(json.dumps(
        {"spmm": {"w1": {"dram_bytes_per_launch": 123, "solver_src_sha1": sha},
                  "w2": {"dram_bytes_per_launch": 456, "solver_src_sha1": "0" * 40}}}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "solver_src_sha1", lambda: sha)
    assert bench._traffic("spmm", "w1") == 123
    assert bench._traffic("spmm", "w2") is None
    assert bench._traffic("spmm", "w3") is None
    assert bench._traffic("cg_resident", "w1") is None


def test_operator_algorithmic_bytes():
    sys.path.insert(0, ROOT)
    import bench

    n, m, kc = 1000, 5000, 64
    unweighted = 4 * 2 * m + 8 * (n + 1) + 2 * 4 * n * kc
    assert bench.spmm_algorithmic_bytes(n, m, kc, False) == unweighted
    assert bench.spmm_algorithmic_bytes(n, m, kc, True) == unweighted + 4 * 2 * m


def test_capped_oracle_sample_keeps_the_contract(monkeypatch, capsys):
    """The sample used on graphs of more than CAPPED_EDGES edges (one column's CG capped, scaled
    to the column's iteration count), exercised on the 2k-node workload."""
    import argparse

    sys.path.insert(0, ROOT)
    import bench

    monkeypatch.setattr(bench, "CAPPED_EDGES", 0)
    args = argparse.Namespace(config="ring_chords_n2000", K=None, steps=2, warmup=1, gpus=1,
                              precond="none")
    bench.run_reference(args, 1, 0)
    d = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert d["impl"] == "reference" and d["value"] > 0 and d["config"]["K"] == 64
    assert "CG iterations" in d["cpu_baseline"]["sample"]
    assert "full oracle solve of column 0" in d["cpu_baseline"]["sample"]
    run = bench.OracleRun("ring_chords_n2000")
    T = run.column_iterations(64)
    v, _, desc, est = bench.oracle_sample_capped(run, 64, T, cap=5)
    assert v > 0 and est > run.t_build and "5 CG iterations" in desc


def test_solve_algorithmic_bytes():
    """The single-launch solvers' bytes: CSR per iteration of the slowest column, 36 bytes per row
    per column-iteration (P, Ap, 7 update passes), initialisation, and the resident kernel's
    true-residual pass."""
    sys.path.insert(0, ROOT)
    import bench

    n, m, kc = 1000, 5000, 4
    iters = [10, 12, 7, 12]
    csr = 4 * 2 * m + 8 * (n + 1)
    expect = 12 * csr + sum(iters) * 36 * n + 12 * n * kc
    assert bench.solve_algorithmic_bytes(n, m, kc, False, iters, False) == expect
    assert bench.solve_algorithmic_bytes(n, m, kc, False, iters, True) == \
        expect + bench.spmm_algorithmic_bytes(n, m, kc, False) + 4 * n * kc
    # a weighted graph reads its CSR weights once per iteration as well
    assert bench.solve_algorithmic_bytes(n, m, kc, True, iters, False) == expect + 12 * 4 * 2 * m
