"""Host logic of bench.py that decides what the bench line reports (no GPU): the committed
DRAM-traffic figure is used only for the kernel source and the workload it was taken on."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_03893_gb300 import synthetic as syn  # noqa: E402


def _read(f):
    return open(os.path.join(ROOT, f), encoding="utf-8").read()


def test_kernel_hash_ignores_comments_and_blank_lines_only():
    h = bench.kernel_hash()
    assert bench.kernel_hash(lambda f: _read(f) + "\n\n// a note\n") == h
    assert bench.kernel_hash(lambda f: _read(f).replace("\n", "\n\n")) == h
    assert bench.kernel_hash(lambda f: _read(f) + "\nint x;\n") != h


def _file_fields():
    kv = {}
    for ln in open(bench.TRAFFIC_FILE):
        if ":" in ln and not ln.startswith("#"):
            a, b = ln.split(":", 1)
            kv[a.strip()] = b.strip()
    return kv


def test_committed_traffic_only_for_its_kernel_and_workload():
    kv = _file_fields()
    w = syn.workload(kv["workload"])
    got = bench.committed_traffic(w)
    if kv["kernel_source_sha256_16"] == bench.kernel_hash():
        assert got == float(kv["dram_bytes_per_launch"])
        assert got == float(kv["captured_dram_bytes"]) * float(kv["scale"])
    else:
        assert got is None
    # a changed field (another kernel instance, or other traffic) or another workload: none
    assert bench.committed_traffic(syn.workload(kv["workload"], weight_dtype="f32")) is None
    assert bench.committed_traffic(syn.workload(kv["workload"], T=4096)) is None
    assert bench.committed_traffic(syn.workload(kv["captured_workload"])) is None


def test_traffic_scale_is_the_token_ratio():
    kv = _file_fields()
    full, cap = syn.workload(kv["workload"]), syn.workload(kv["captured_workload"])
    assert float(kv["scale"]) == full.n_tokens / cap.n_tokens
    # the per-launch figure stays close to the algorithmic bytes of the full launch
    alg = bench.algorithmic(full)["bytes"]
    assert 0.95 * alg < float(kv["dram_bytes_per_launch"]) < 1.10 * alg


def test_no_reuse_bound_has_the_stated_intensity():
    # per head: each (target layer, K|V, head) product reads k tiles of d channels and
    # writes d, 2 k d d FLOP per token: intensity k d / (k + 1)
    for name in ("qwen3_14b_32b_t32768_k4", "qwen3_14b_32b_t32768_k1", "llama31_8b_70b_b4x8192_k3"):
        w = syn.workload(name)
        alg = bench.algorithmic(w)
        assert alg["no_reuse_intensity"] == w.k * w.d / (w.k + 1)
        # reuse only lowers the bytes: source once and target once
        assert alg["no_reuse_bytes_per_token"] >= alg["bytes_per_token"] - 4
    # cross-head: one product per (target layer, K|V) reads k H d features and writes H d,
    # 2 (k H d) (H d) FLOP per token: intensity k H d / (k + 1)
    w = syn.workload("qwen3_14b_32b_t32768_k4_xhead")
    alg = bench.algorithmic(w)
    assert alg["no_reuse_intensity"] == w.k * w.H * w.d / (w.k + 1)
    peaks = {"bf16": 1900.0, "hbm": 6800.0}
    b = bench.no_reuse_bound(bench.algorithmic(syn.workload("qwen3_14b_32b_t32768_k4")),
                             syn.workload("qwen3_14b_32b_t32768_k4"), peaks, 3.0)
    # 1024 products x (512 + 128) x 2 B = 1,310,720 B per token; over 32768 tokens at
    # 6.8 TB/s that is 6.316 ms, above the 2.315 ms of FLOPs; frac is bound time / measured
    assert b["bytes_per_token"] == 1310720
    assert b["bound"] == "hbm" and abs(b["roofline_ms"] - 32768 * 1310720 / 6.8e9) < 1e-9
    assert abs(b["frac"] - b["roofline_ms"] / 3.0) < 1e-12


def test_algorithmic_counts_of_the_workloads():
    """Per launch, as stated for the bench workloads: FLOP = 2 (K, V) L_t H 2 F d per token;
    bytes = every source layer read once + the target written once + 4 B of position per
    token, plus W and b once."""
    w = syn.workload("qwen3_14b_32b_t32768_k4")
    a = bench.algorithmic(w)
    assert a["flop"] == 4_398_046_511_104 and a["flop_per_token"] == 134_217_728
    assert a["bytes_per_token"] == 163_840 + 262_144 + 4
    assert a["weight_bytes"] == 134_217_728 + 262_144                 # W bf16, then b
    assert a["bytes"] == 14_093_254_656
    # Llama-3.1 8B -> 70B shapes: more target than source layers, k = 3
    a = bench.algorithmic(syn.workload("llama31_8b_70b_b4x8192_k3"))
    assert a["flop"] == 4_123_168_604_160
    assert a["bytes_per_token"] == 131_072 + 327_680 + 4
    assert a["weight_bytes"] == 125_829_120 + 327_680
    assert a["bytes"] == 15_158_673_408
    # fp32 caches and weights count 4 bytes an element; fp32 weights on bf16 caches too
    w = syn.workload("tiny_fp32")
    a = bench.algorithmic(w)
    assert a["bytes_per_token"] == 2 * 4 * 2 * 64 * 4 + 2 * 6 * 2 * 64 * 4 + 4
    assert a["weight_bytes"] == (6 * 2 * 2 * 128 * 64 + 6 * 2 * 2 * 64) * 4
    a = bench.algorithmic(syn.workload("qwen3_14b_32b_t32768_k4", weight_dtype="f32"))
    assert a["bytes_per_token"] == 163_840 + 262_144 + 4 and a["weight_bytes"] == 2 * (134_217_728 + 262_144)
    # one paged turn (16 x 2048 new tokens), Qwen3-32B -> 14B shapes
    a = bench.algorithmic(syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4"))
    assert a["flop"] == 2_748_779_069_440 and a["bytes_per_token"] == 262_144 + 163_840 + 4


class _Clocks(bench.ClockSampler):
    def __init__(self, out):
        super().__init__(0)
        self.out = out


def test_clock_summary():
    # index, clocks.sm, clocks.max.sm, power.draw, reasons.active, hw, hw_thermal, sw_thermal, sw_power_cap
    rows = ["0, 1980, 2070, 150.0, 0x0, Not Active, Not Active, Not Active, Not Active",   # idle: not under load
            "0, 1500, 2070, 1390.0, 0x4, Not Active, Not Active, Not Active, Active",
            "0, 1700, 2070, 1200.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            "0, 1600, 2070, 1300.5, 0x0, Not Active, Not Active, Not Active, Not Active",
            "0, 1650, 2070, 1250.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            "garbage line", "0, [N/A], 2070, 900, 0x0, Not Active, Not Active, Not Active, Not Active"]
    s = _Clocks("\n".join(rows)).summary()
    assert s["sm_mhz"] == 1625.0                     # median of the four loaded samples
    assert s["sm_max_mhz"] == 2070.0 and s["reasons"] == ["sw_power_cap"]
    assert s["samples"] == 5 and s["samples_under_load"] == 4 and s["power_w_max"] == 1390.0
    hot = rows[1].replace("Not Active, Not Active, Not Active, Active", "Active, Not Active, Active, Not Active")
    assert _Clocks(hot).summary()["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]
    hot = rows[1].replace("Not Active, Not Active, Not Active, Active", "Not Active, Active, Not Active, Not Active")
    assert _Clocks(hot).summary()["reasons"] == ["hw_thermal_slowdown"]
    # below 200 W everywhere: every sample counts; no samples at all: said so
    idle = _Clocks(rows[0] + "\n" + rows[0].replace("1980", "1000")).summary()
    assert idle["sm_mhz"] == 1490.0 and idle["samples_under_load"] == 2
    assert _Clocks("").summary() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"]}
    # under load means above 200 W; the maximum clock is the largest reported
    edge = ["0, 1000, 1980, 200.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            "0, 1800, 2070, 200.05, 0x0, Not Active, Not Active, Not Active, Not Active",
            "0, 1900, 2010, 600.0, 0x0, Not Active, Not Active, Not Active, Not Active"]
    e = _Clocks("\n".join(edge)).summary()
    assert e["samples_under_load"] == 2 and e["sm_mhz"] == 1850.0 and e["sm_max_mhz"] == 2070.0


def test_peaks_fallback_is_the_recipe_figures(monkeypatch, tmp_path):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.load_peaks() == dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, source="fallback")
    (tmp_path / "MEASURED_PEAKS.json").write_text('{"hbm_gbs": 6000.5, "bf16_tflops": 1800.25}')
    assert bench.load_peaks() == dict(hbm=6000.5, bf16=1800.25, bf16_sustained=None, source="measured")


def test_traffic_file_parsing(monkeypatch, tmp_path):
    w = syn.workload("qwen3_14b_32b_t32768_k4")
    f = tmp_path / "traffic.txt"
    f.write_text("# a comment: kernel_source_sha256_16: 0000000000000000\n"
                 "# workload: elsewhere\n"
                 "\n"
                 "a line of text\n"
                 "kernel_source_sha256_16: %s\nworkload: %s\ncaptured_workload: x:y\n"
                 "dram_bytes_per_launch: 123456789\n" % (bench.kernel_hash(), w.name))
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(f))
    assert bench.committed_traffic(w) == 123456789.0
    f.write_text("kernel_source_sha256_16: %s\nworkload: %s\ndram_bytes_per_launch: n/a\n" % (bench.kernel_hash(), w.name))
    assert bench.committed_traffic(w) is None


def test_reference_arm_prints_the_contract_line(capsys):
    import json
    import types
    w = syn.workload("tiny_fp32")
    args = types.SimpleNamespace(steps=3, warmup=1, gpus=1)
    config = {"workload": w.name}
    assert bench.reference_arm(args, w, config) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC and line["unit"] == bench.UNIT
    assert (line["n_gpus"], line["steps"], line["warmup"]) == (1, 3, 1)
    assert line["higher_is_better"] is True and line["vs_baseline"] is None and line["dtype"] == "f64"
    assert line["config"] == config and line["value"] > 0 and line["ms_per_step"] > 0
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == line["value"] and cb["unit"] == line["unit"] and cb["cores"] >= 1
    assert "tokens" in cb["sample"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
