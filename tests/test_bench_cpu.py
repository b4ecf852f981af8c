"""Host-side parts of bench.py on the CPU: the reference arm (the oracle timed
on the host cores) prints one well-formed JSON line, and fanning the oracle's
attention out over threads by row chunks returns exactly what one call over
the same rows returns (each row is computed on its own); the DRAM-traffic
records follow the attention code, not its comments."""
import json
import os
import subprocess
import sys

import numpy as np

import oracle
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "1"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "steps/s" and line["higher_is_better"] is True
    assert line["value"] > 0 and line["steps"] == 2 and line["warmup"] == 1
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"]
    ex = line["extrapolated"]
    assert 1 <= ex["rows_timed"] <= ex["rows_total"] and abs(ex["scale"] - ex["rows_total"] / ex["rows_timed"]) < 1e-9
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]


def test_threaded_oracle_attention_equals_one_call():
    sys.path.insert(0, ROOT)
    import bench
    w = synth.build(synth.small_spec(B=3, V=300), seed=4)
    s = w.spec
    rows = [(n, h) for n in range(w.R) for h in range(s.Hq)]
    one = oracle.tree_attn(w.q, w.k, w.v, w.kv_off, w.ctx_len, w.node_off, w.parents, s.Hq, s.Hkv, s.D,
                           s.D ** -0.5, rows=rows)
    # the test helper's fan-out (row chunks over threads, results concatenated)
    sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))
    import gpu_helpers
    fan = gpu_helpers.oracle_attn(w, s.D ** -0.5, rows=None, workers=4)
    assert (fan["rows"] == one["rows"]).all()
    assert np.array_equal(fan["out"], one["out"]) and np.array_equal(fan["lse"], one["lse"])
    # the benchmark's fan-out runs the same rows (it only times them)
    bench.oracle_attn_rows(w, rows[:17], workers=4)
    assert bench.host_cores() >= 1


def test_traffic_records_follow_the_code_not_the_comments(tmp_path, monkeypatch):
    # the committed DRAM-traffic records are keyed by a hash of the attention
    # sources with comments and blank space taken out: a comment edit keeps
    # them, any change to the code retires them
    sys.path.insert(0, ROOT)
    import bench
    csrc = tmp_path / "paper_2511_01282_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in ("attn.cu", "attn_core.cuh", "attn_pair.cuh", "sm100.cuh"):
        (csrc / f).write_text(open(os.path.join(ROOT, "paper_2511_01282_gb300", "csrc", f)).read())
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.attn_source_sha()
    core = csrc / "attn_core.cuh"
    src = core.read_text()
    core.write_text(src.replace("namespace rs {", "// a new comment line\nnamespace rs {  /* and a block */", 1))
    assert bench.attn_source_sha() == h0
    core.write_text(src.replace("constexpr int kNS = 3;", "constexpr int kNS = 4;", 1))
    assert bench.attn_source_sha() != h0
