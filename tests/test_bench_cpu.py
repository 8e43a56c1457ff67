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
