"""bench.py's command-line contract on a host without a GPU: the reference arm (the
float64 oracle on the host cores) prints one well-formed JSON line, and our arm fails
loudly instead of falling back to the CPU."""
import json
import os
import subprocess
import sys

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(*args, timeout=600):
    env = dict(os.environ, OMP_NUM_THREADS=os.environ.get("OMP_NUM_THREADS", "4"))
    return subprocess.run([sys.executable, "bench.py", *args], cwd=ROOT, env=env, capture_output=True, text=True,
                          timeout=timeout)


def test_reference_arm_prints_one_json_line():
    p = _run("--impl", "reference", "--steps", "1", "--warmup", "1")
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [ln for ln in p.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    assert (d["n_gpus"], d["steps"], d["warmup"]) == (1, 1, 1)
    assert d["unit"] == "tok/s" and d["higher_is_better"] is True and d["vs_baseline"] is None
    assert d["value"] > 0 and d["ms_per_step"] > 0
    M = d["config"]["M"]
    assert d["value"] * d["ms_per_step"] == pytest.approx(1e3 * M, rel=1e-9)
    assert "workload" in d["config"] and d["dtype"] == "f64" and d["scaling"] == "weak"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "tok/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the behaviour without a GPU")
def test_our_arm_fails_loudly_without_a_gpu():
    p = _run("--steps", "1", "--warmup", "3", timeout=300)
    assert p.returncode != 0
    assert not [ln for ln in p.stdout.splitlines() if ln.startswith("{")]


def _bench_module():
    import importlib.util

    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    b = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(b)
    return b


def test_traffic_staleness_hash_follows_the_kernel_sources(tmp_path):
    """The committed ncu traffic stays valid across host-only edits, comment edits and new
    function prototypes in the public headers, and is dropped once a source of the kernel
    itself, or a type or constant of the headers, changes."""
    import shutil

    b = _bench_module()
    for d in ("paper_2405_03594_gb300/csrc", "include"):
        shutil.copytree(os.path.join(ROOT, d), tmp_path / d)
    b.ROOT = str(tmp_path)
    base = {k: b.kernel_source_hash(k) for k in b.KERNEL_SOURCES}
    assert b.kernel_source_hash("no_such_kernel") is None

    def edit(rel, old, new):
        p = tmp_path / rel
        s = p.read_text()
        assert old in s
        p.write_text(s.replace(old, new, 1))

    edit("paper_2405_03594_gb300/csrc/sp_api.cu", "extern \"C\" {", "extern \"C\" {\n// host-only edit")
    edit("include/sp.h", "/*", "/* comment edit;")
    edit("include/sp.h", "#ifdef __cplusplus\n}", "sp_status sp_new_entry(const sp_matrix* h,\n  int64_t m);\n"
         "#ifdef __cplusplus\n}")
    assert {k: b.kernel_source_hash(k) for k in b.KERNEL_SOURCES} == base
    edit("paper_2405_03594_gb300/csrc/sp_linear_tc.cu", "namespace sp {", "namespace sp {\nstatic int edited;")
    now = {k: b.kernel_source_hash(k) for k in b.KERNEL_SOURCES}
    assert now["linear_tc_kernel"] != base["linear_tc_kernel"]
    assert all(now[k] == base[k] for k in base if k != "linear_tc_kernel")
    edit("include/sp.h", "#define", "#define SP_EDITED 1\n#define")
    assert all(b.kernel_source_hash(k) != base[k] for k in base)
    mid = {k: b.kernel_source_hash(k) for k in b.KERNEL_SOURCES}
    edit("include/sp.h", "SP_ERR_WORKSPACE = 8", "SP_ERR_WORKSPACE = 9")
    assert all(b.kernel_source_hash(k) != mid[k] for k in base)


def test_committed_traffic_matches_the_current_kernel_sources():
    """Each committed ncu traffic figure carries the hash of the sources it was taken on;
    those that still match the current sources are the ones the bench reports."""
    b = _bench_module()
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        d = json.load(f)
    for key, e in d.items():
        kernel, workload = key.split("|", 1)
        assert kernel in b.KERNEL_SOURCES and e["dram_bytes_per_launch"] > 0
        got = b.profiled_traffic(kernel, workload)
        assert got == (e["dram_bytes_per_launch"] if e["source_hash"] == b.kernel_source_hash(kernel) else None)


def test_cpu_baseline_leg_runs_the_oracle_for_the_requested_time():
    """The bench's cpu_baseline: the float64 oracle on the host cores, repeated for about
    the requested time (at least three runs), scaled to a full step."""
    import time

    import numpy as np

    b = _bench_module()
    g = np.random.default_rng(0)
    host = {}
    for name in b.SHAPES:
        N, K = 40, 64
        W = g.standard_normal((N, K)).astype(np.float32)
        host[name] = (b.np.asarray(W.view(np.uint32) >> 16, dtype=np.uint16),
                      (g.random((N, K)) < 0.3).astype(np.uint8),
                      np.zeros((2, K), dtype=np.uint16))
    t0 = time.perf_counter()
    cb, outs = b.cpu_oracle_leg(host, 1, reps_target_s=0.3)
    assert time.perf_counter() - t0 >= 0.3
    assert cb["kind"] == "oracle" and cb["unit"] == "tok/s" and cb["cores"] >= 1 and cb["value"] > 0
    runs = int(cb["sample"].split("median of ")[1].split()[0])
    assert runs >= 3
    assert set(outs) == set(b.SHAPES) and all(outs[n].shape == (1, 40) for n in b.SHAPES)
    assert all(not outs[n].any() for n in b.SHAPES)  # x = 0 gives y = 0


def test_dense_section_reports_failures_instead_of_raising():
    """The dense cuBLAS comparison is context: on a host without a GPU it returns its
    failure inside the section (with the paper's quoted speedups) rather than raising."""
    b = _bench_module()
    out = b.dense_section({}, {}, {}, [1])
    assert "error" in out and out["paper"]["gpu_sparsity_only"]["x"] == 1.7
    assert out["shapes"] == {} and out["step_speedup"] == {}


def test_update_bytes_counts_gradient_sectors_values_masks_and_offsets():
    """Roofline bytes of one masked update, by hand: a 128 x 64 matrix (one chunk) whose
    row 0 keeps columns 0 and 9 and row 1 keeps column 63: gradient sectors of 8 columns
    holding a kept column are (0, 0), (0, 1) and (1, 7), so 3 x 32 bytes; 3 kept values are
    read and written (3 x 4 bytes); the masks are 128 x 64 / 8 bytes; 2 chunk offsets."""
    import numpy as np

    b = _bench_module()
    mask = np.zeros((128, 64), dtype=np.uint8)
    mask[0, 0] = mask[0, 9] = mask[1, 63] = 1

    class Info:
        nnz, tiles, row_blocks = 3, 1, 1

    assert b.update_bytes(mask, Info) == 3 * 32 + 3 * 4 + 128 * 64 // 8 + 2 * 8


def test_update_section_reports_failures_instead_of_raising():
    """The masked-update section is context next to the decode step: without a GPU it
    returns its failure inside the section rather than ending the run."""
    b = _bench_module()
    out = b.update_section(None, {n: (None, None, None) for n in b.SHAPES}, 6681.8)
    assert "error" in out and out["shapes"] == {} and out["kernel"] == "masked_update_kernel"


def test_sweep_copies_exceed_three_l2():
    """A graph over the sweep's copies reads more than 3x L2 of distinct compressed bytes."""
    b = _bench_module()
    for nbytes in (10_000_000, 45_000_000, 65_400_000, 191_600_000, 500_000_000):
        c = b.sweep_copies(nbytes)
        assert c * nbytes > 3 * b.L2_BYTES  # enough copies
        assert c == 2 or (c - 1) * nbytes <= 3 * b.L2_BYTES  # and no more than needed (at least 2)


def test_roofline_time_takes_the_slower_bound():
    """Bytes over HBM peak against nonzero FLOPs over tensor peak, by hand: 66.2 MB at
    6681.8 GB/s is 9.907 us; 2 * 256 * 27e6 FLOPs at 1936.4 TFLOP/s is 7.14 us (HBM-bound),
    and at M = 2048 the FLOPs (57.1 us) win."""
    b = _bench_module()
    t, bound = b.roofline_time_us(66_200_000, 27_000_000, 256, 6681.8, 1936.4)
    assert bound == "hbm" and t == pytest.approx(66.2e6 / 6681.8e9 * 1e6)
    t, bound = b.roofline_time_us(66_200_000, 27_000_000, 2048, 6681.8, 1936.4)
    assert bound == "tensor" and t == pytest.approx(2 * 2048 * 27e6 / 1936.4e12 * 1e6)


def test_sweep_section_reports_failures_instead_of_raising():
    b = _bench_module()
    out = b.sweep_section(None, 6681.8)
    assert "error" in out and out["points"] == {}


def _full_sections():
    """Context sections shaped like a full run's (every shape, sparsity and batch size)."""
    per_shape = {n: {"us_per_launch": 24.41234, "gbs": 2680.51234, "frac": 0.401234} for n in ("qkv", "o", "gate_up",
                                                                                                 "down")}
    per_m = {str(m): {"tok_s": 445.928809 * m, "step_ms": 2.242510414, "step_gbs": 2095.73218, "frac_of_peak": 0.3136,
                      "per_shape": {n: {"us": 1.0, "gbs": 2.0, "frac": 0.3} for n in per_shape}} for m in (1, 4, 16)}
    by_m = {str(m): {"us": 31.5, "tok_s": 1.0, "gbs": 765.97, "tflops_nonzero": 9.15, "bound": "hbm",
                     "frac_of_roofline": 0.1146353276, "kernel": "linear_tc_kernel"} for m in (1, 2, 4, 8, 16, 32, 64,
                                                                                               128, 256)}
    return {
        "per_m": per_m,
        "chained_step_bf16": {"chain": {"1": {"tok_s": 420.123456}, "4": {"tok_s": 1229.98765}},
                              "graph": {"1": {"tok_s": 430.111}, "4": {"tok_s": 1350.222}}},
        "stack_int8": {"graph_per_m": {"1": {"tok_s": 355.1234}, "16": {"tok_s": 2902.123}, "64": {"tok_s": 9684.1}},
                       "chain_per_m": {"1": {"tok_s": 368.12}, "4": {"tok_s": 1048.4}}},
        "prefill": {"shapes": {f"{n}@{p}%": {"frac_dense_executed": 0.3212345} for n in per_shape for p in (50, 70)}},
        "masked_update": {"shapes": {n: {"frac": 0.4612345} for n in per_shape}},
        "w8a8": {"shapes": {n: {str(m): {"w8a8_over_int8_weight": 1.2345678} for m in (1, 16, 64)}
                            for n in ("gate_up", "down")}},
        "dense_comparison": {"step_speedup": {"1": 2.3456789, "4": 2.1, "16": 1.9}},
        "sparsity_batch_sweep": {"points": {f"{n}@{p}%": {"by_m": by_m} for n in ("gate_up", "down")
                                            for p in (0, 50, 60, 70, 80)}},
        "per_layer_profile": {"chain": {"tok_s": 431.12345}, "graph": {"tok_s": 440.12345}},
        "square_12288": {"points": {str(p): {"speedup_vs_0pct": 1.23456789} for p in range(0, 100, 10)}},
    }


def test_headline_line_is_compact_and_complete():
    """The final stdout line must survive a tail capture whole: about 2 KB at most with
    every context section present, and carrying every key of the bench contract."""
    import argparse

    b = _bench_module()
    args = argparse.Namespace(m=1, pct=70, path="auto", steps=20, warmup=5)
    r = {"tok_s": 445.92880982, "step_ms": 2.2425104141, "step_gbs": 2095.732184, "step_bytes": 4_700_000_000}
    roofline = {"bound": "hbm", "achieved": 2680.5123, "peak": 6681.8, "unit": "GB/s", "frac": 0.40116,
                "traffic": 65_930_000, "kernel": "linear_ccw_kernel", "launch": "gate_up 70% bf16 M=1",
                "peak_kind": "of measured",
                "algorithmic_bytes_per_launch": 65_440_000, "us_per_launch": 24.41234,
                "frac_of_nominal_8tbs": 0.3350123}
    e2e = {"value": 422.123456789, "unit": "tok/s", "h2d_bytes_per_step": 8192 * 4 + 22016, "d2h_bytes_per_step": 8192}
    cpu = {"value": 1.1812345, "unit": "tok/s", "cores": 16, "kind": "oracle",
           "sample": "layer 0 (qkv, o, gate_up, down) at M=1, float64 C oracle, OpenMP over rows; "
                     "median of 12 runs of 0.85 s, x32 layers"}
    clocks = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 123}
    parity = {"max_err_over_max_ref": 0.00212345, "rel_fro": 0.00112345, "ok": True}
    line = b.headline_line(args, 1, r, roofline, e2e, cpu, clocks, parity, 20 * 128,
                           b.section_summary(_full_sections()))
    text = json.dumps(line, separators=(",", ":"))  # as bench.py prints it
    assert len(text) <= 2048, len(text)
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "e2e", "gpu_launches", "roofline", "cpu_baseline", "clocks"):
        assert k in line, k
    assert line["config"]["workload"] and line["roofline"]["frac"] == pytest.approx(0.4012, abs=1e-4)
    assert line["value"] == pytest.approx(445.929, rel=1e-5)
    assert set(line["summary"]["sweep_frac"]) == {"gate_up@70%", "down@70%"}
    assert set(line["summary"]["square_speedup_vs_0pct"]) == {"50", "70", "90"}
    assert line["summary"]["profile_tok_s"]["chain"] == pytest.approx(431.1, abs=0.1)
    assert "errors" not in line["summary"]


def test_section_summary_reports_section_errors():
    b = _bench_module()
    s = b.section_summary({"prefill": {"error": "RuntimeError: " + "x" * 500, "shapes": {}}})
    assert s["errors"]["prefill"].startswith("RuntimeError") and len(s["errors"]["prefill"]) <= 80


def test_profile_and_square_sections_report_failures_instead_of_raising():
    """The per-layer profile and 12K x 12K sections are context: without a GPU they return
    their failure inside the section rather than ending the run."""
    import argparse

    b = _bench_module()
    args = argparse.Namespace(steps=3, warmup=3)
    pr = b.profile_section(args, 6681.8)
    assert "error" in pr and sum(pr["profile"]) == 70 * b.LAYERS
    sq = b.square_section(args)
    assert "error" in sq and sq["points"] == {}


def test_kernel_source_hash_ignores_comments_but_not_code(tmp_path, monkeypatch):
    """The traffic record stays valid across comment edits of a kernel's sources and is
    discarded by any code edit."""
    import shutil

    b = _bench_module()
    root = tmp_path / "repo"
    shutil.copytree(os.path.join(b.ROOT, "paper_2405_03594_gb300", "csrc"), root / "paper_2405_03594_gb300" / "csrc")
    shutil.copytree(os.path.join(b.ROOT, "include"), root / "include")
    monkeypatch.setattr(b, "ROOT", str(root))
    base = b.kernel_source_hash("linear_ccw_kernel")
    src = root / "paper_2405_03594_gb300" / "csrc" / "sp_linear_cc.cu"
    text = src.read_text()
    src.write_text("// a new comment line\n" + text.replace("// Launch:", "/* block comment */ // Launch:", 1))
    assert b.kernel_source_hash("linear_ccw_kernel") == base
    src.write_text(text.replace("constexpr int kCtasPerSm = 4;", "constexpr int kCtasPerSm = 5;", 1))
    assert b.kernel_source_hash("linear_ccw_kernel") != base
