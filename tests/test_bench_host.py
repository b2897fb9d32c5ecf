"""Host-side pieces of bench.py that need no GPU: the DRAM-traffic ratio taken from the
committed ncu summary (and dropped once the profiled kernel source changes), and the
clock/throttle summary parsed from nvidia-smi samples."""
import hashlib
import os

import bench
from paper_2607_12287_gb300 import synth

GEMM_SRC = os.path.join(bench.ROOT, "paper_2607_12287_gb300", "csrc", "gemm.cu")


def _tree(tmp_path, src: str, ratio: float, digest: str):
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "gemm_tc_kernel_so400m_224_1view.md").write_text(
        f"traffic_to_algorithmic_ratio: {ratio}\ngemm_tc_kernel_source_sha256: {digest}\n")
    csrc = tmp_path / "paper_2607_12287_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "gemm.cu").write_text(src)


def test_traffic_ratio_follows_the_profiled_source(tmp_path, monkeypatch):
    src = open(GEMM_SRC).read()
    cut = src.find("// Many-tile form")
    assert cut > 0
    digest = hashlib.sha256(src[:cut].encode()).hexdigest()
    _tree(tmp_path, src, 0.99, digest)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.gemm_traffic_ratio() == 0.99
    # a change below the profiled kernel (the warp-specialised form) keeps the ratio
    (tmp_path / "paper_2607_12287_gb300" / "csrc" / "gemm.cu").write_text(src + "\n// tail\n")
    assert bench.gemm_traffic_ratio() == 0.99
    # a change inside the profiled kernel drops it
    (tmp_path / "paper_2607_12287_gb300" / "csrc" / "gemm.cu").write_text("// edit\n" + src)
    assert bench.gemm_traffic_ratio() is None


def test_traffic_ratio_absent_summary(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.gemm_traffic_ratio() is None


def test_clock_summary_parses_samples_and_reasons(tmp_path):
    csv = tmp_path / "clocks.csv"
    csv.write_text(
        "0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active\n"
        "0, 2055, 2070, 1390.5, 0x4, Not Active, Not Active, Not Active, Active\n"
        "0, 2070, 2070, 1201.0, 0x0, Not Active, Not Active, Not Active, Not Active\n"
        "garbage line\n")
    s = bench.ClockSampler(0)
    s.proc, s.path = object(), str(csv)  # as if nvidia-smi had written the file
    out = s.summary()
    assert out == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "samples": 3, "reasons": ["sw_power_cap"]}
    assert not csv.exists()  # the sample file is removed once read


def test_clock_summary_without_nvidia_smi():
    s = bench.ClockSampler(0)
    assert s.summary() is None


def test_describe_names_the_workload():
    from paper_2607_12287_gb300 import synth
    d = bench.describe(synth.WORKLOADS["so400m_224_1view"])
    assert d["workload"] == "so400m_224_1view" and d["views"] == 1
    assert "dim 1152" in d["encoder"] and "27 layers" in d["encoder"]
    assert bench.describe(synth.sweep_workload(0.25))["selection"] == "top-64"


def test_algorithmic_bytes_per_step_so400m():
    # weights 823.5 MB of bf16 matrices + 27 layers of cached K/V (31.9 MB) + frame +
    # embeddings + the updated rows' writes: about 0.86 GB for the 1-view 224 px stream
    import bench
    wl = synth.WORKLOADS["so400m_224_1view"]
    w = bench.weight_matrix_bytes(wl.shape)
    assert abs(w - 823.5e6) < 1.5e6
    b = bench.algorithmic_bytes_per_step(wl, 26)
    assert 0.85e9 < b < 0.87e9
    assert bench.algorithmic_bytes_per_step(wl, 52) > b


def test_ideal_speedup_follows_the_roofline():
    # One 224 px So400m view: both calls stream the same 824 MB of weights and the full
    # encode's 220 GFLOP take as long at the tensor peak, so a perfect implementation
    # gains nothing from skipping rows (ratio ~1).  Three views with 5/15/30% updated rows
    # share the weights across three views' worth of full-encode FLOPs: about 2.7.
    pk = {"hbm_gbs": 6785.5, "bf16_tflops_sustained": 1716.2}
    one = synth.WORKLOADS["so400m_224_1view"]
    inc = bench.ideal_ms_per_step(one, 0.1 * 256, False, pk)
    full = bench.ideal_ms_per_step(one, 0.1 * 256, True, pk)
    assert inc["bound"] == "hbm" and full["bound"] == "tensor"
    assert 0.95 < full["ms"] / inc["ms"] < 1.05
    # the full encode's FLOPs: 2 * params-per-token * tokens plus attention, per layer
    s = one.shape
    per_row = 2.0 * (4 * s.dim * s.dim + 2 * s.dim * s.mlp_dim) + 4.0 * s.n_tokens * s.dim
    embed = 2.0 * s.n_tokens * s.dim * s.patch * s.patch * 3
    assert abs(full["flops"] - (embed + s.depth * s.n_tokens * per_row)) < 1e-6 * full["flops"]
    three = synth.WORKLOADS["so400m_224_3view"]
    rows = 256 * (0.05 + 0.15 + 0.30)
    r3 = bench.ideal_ms_per_step(three, rows, True, pk)["ms"] / bench.ideal_ms_per_step(three, rows, False, pk)["ms"]
    assert 2.5 < r3 < 2.9
