"""The bench's reference arm and its JSON line (CPU): `bench.py --impl
reference` times the oracle on the measured arm's workload config, metric and
unit and prints one line with the keys the measurement contract asks for."""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def run_bench(*args):
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args],
                         cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, out.stdout[-2000:]
    return json.loads(lines[0])


def test_default_workload_is_the_largest_single_gpu_config():
    import bench
    import synth

    w = synth.WORKLOADS[bench.DEFAULT_WORKLOAD]
    hbm = [x for x in synth.WORKLOADS.values()
           if x.location == "device" and x.B * x.L > 0 and x.d > 8]
    assert w.n_fgrams * w.d == max(x.n_fgrams * x.d for x in hbm)


def test_reference_line_keys():
    import bench

    # the tiny workload keeps this CPU test short; the default (large_hbm)
    # runs the same code on a larger batch
    d = run_bench("--impl", "reference", "--workload", "tiny", "--steps", "2", "--warmup", "1")
    assert d["impl"] == "reference"
    assert d["metric"] == bench.METRIC and d["unit"] == "tokens/s"
    assert d["higher_is_better"] is True and d["value"] > 0
    assert d["warmup"] >= 3 and d["steps"] == 2
    import synth

    w = synth.WORKLOADS["tiny"]
    # the arm times what its config names: one whole B x L batch per step
    assert d["config"]["workload"] == bench.prefill_config(w, 1)["workload"]
    assert d["config"]["global_batch_tokens"] == w.B * w.L
    assert f"{w.B} x {w.L}" in d["cpu_baseline"]["sample"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] == 1 and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_reference_line_other_workload_is_explicit():
    d = run_bench("--impl", "reference", "--workload", "discover", "--steps", "1")
    assert d["impl"] == "reference" and "unavailable" in d


def test_kernel_names_and_profile_lookup():
    """The roofline's kernel follows the launch the copy mode and the table's
    suffix index select, and a profile summary counts only while its source
    hash matches the current sources."""
    import bench

    assert bench.embed_kernel_name("auto", 3, True).startswith("embed_walk_kernel")
    assert bench.embed_kernel_name("auto", 5, True).startswith("embed_walk_kernel")
    assert bench.embed_kernel_name("auto", 5, False).startswith("embed_pipe_kernel")
    assert bench.embed_kernel_name("auto", 3, False).startswith("embed_kernel")
    assert bench.embed_kernel_name("registers", 3, True).startswith("embed_kernel")
    assert bench.embed_kernel_name("pipelined", 3, True).startswith("embed_walk_kernel")
    assert bench.embed_kernel_name("split", 5, True).startswith("embed_split_kernel")
    # the committed summaries of the bench's kernels were taken on these sources
    for wl in ("large_hbm", "stress_k5", "prefill_1b"):
        t, note = bench.profiled_traffic(wl, "embed_walk_kernel", bench.PIPE_SOURCES,
                                         with_note=True)
        assert t is not None and t > 0, wl
    assert bench.profiled_traffic("mixed_serving", "varlen_walk_kernel",
                                  bench.VARLEN_SOURCES) is not None
    # an unknown summary reads as no traffic
    assert bench.profiled_traffic("no_such_workload", "embed_walk_kernel",
                                  bench.PIPE_SOURCES) is None
