#!/usr/bin/env python3
"""Throughput bench for the cross-model KV mapper (one JSON line on rank 0).

Metric: mapped target-KV tokens/s (one token = every target layer x KV head x K and V
written) on the Qwen3-14B->32B-shaped long-context workload: 40 -> 64 layers, 8 KV heads,
head_dim 128, bf16, one sequence of 32768 tokens at positions 0..32767, k = 4 selected
source layers per target layer.  A step is one kvx_map call over the whole workload.

* value: device throughput, inputs resident in HBM, K steps timed with CUDA events on
  the launching stream between a barrier + synchronize on both sides (max over ranks).
  Every step reads 5.4 GB of source cache and writes 8.6 GB of target cache, far more
  than the 129 MB L2, so no flush is needed between steps.
* e2e: the same metric through the C ABI with host buffers: each step copies the source
  caches and positions from pinned host memory, maps, and copies the target cache back.
* roofline: algorithmic FLOPs and bytes of one launch (tensor-core and HBM bounds)
  against MEASURED_PEAKS.json; traffic from the committed ncu summary when it was taken
  on the current kernel source.
* cpu_baseline: the float64 oracle on a bounded sample of the same workload's tokens.
* --impl reference: the oracle as the reference arm.

Multi-GPU (torchrun): every rank maps its own replica (weak scaling, no collective on
the data path; a MAX all-reduce of the elapsed time only).
"""
import argparse
import dataclasses
import hashlib
import re
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_03893_gb300 import kvx  # noqa: E402
from paper_2608_03893_gb300 import synthetic as syn  # noqa: E402

METRIC = "mapped target-KV tokens/s"
UNIT = "tokens/s"
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "tc_map_kernel_qwen3_14b_32b_traffic.txt")
KERNEL_SOURCES = ["paper_2608_03893_gb300/csrc/kvx_tc.cu", "paper_2608_03893_gb300/csrc/kvx_rope.cuh",
                  "paper_2608_03893_gb300/csrc/kvx_internal.h", "paper_2608_03893_gb300/csrc/kvx_ptx.cuh"]


def algorithmic(w):
    """FLOPs and bytes of one launch (per-unit figures times the tokens of the launch).
    Caches count at their element size (bf16 2 bytes, fp32 4), W and b at the weights'
    (fp32 weights are 4 bytes an element, as the bf16 hi + lo pair the kernels read)."""
    e = 4 if w.cache_dtype == "f32" else 2
    ew = 4 if w.weight_dtype == "f32" else 2
    tok = w.n_tokens
    flop_per_tok = 2 * w.Lt * w.H * 2 * w.F * w.d              # K and V contractions
    src_per_tok = 2 * w.Ls * w.H * w.d * e                       # every source layer read once
    tgt_per_tok = 2 * w.Lt * w.H * w.d * e                       # target written once
    w_bytes = w.Lt * 2 * w.H * w.F * w.d * ew + w.Lt * 2 * w.H * w.d * ew
    # looser bound: a mapper without reuse reads the k selected source tiles again for
    # every (target layer, K|V, head) product (per head; one product per (target layer,
    # K|V) cross-head) and writes its output: intensity k d / (k + 1) FLOP per byte per head
    per_head = w.head_mix != "cross_head"
    gemms, out = (2 * w.Lt * w.H, w.d) if per_head else (2 * w.Lt, w.H * w.d)
    no_reuse_per_tok = gemms * (w.F + out) * e
    return dict(flop=flop_per_tok * tok, bytes=(src_per_tok + tgt_per_tok + 4) * tok + w_bytes,
                flop_per_token=flop_per_tok, bytes_per_token=src_per_tok + tgt_per_tok + 4,
                weight_bytes=w_bytes, no_reuse_bytes_per_token=no_reuse_per_tok,
                no_reuse_intensity=flop_per_tok / no_reuse_per_tok)


def no_reuse_bound(alg, w, peaks, ms_step):
    """The roofline of a mapper that re-reads its source tiles for every product (the
    looser bound, intensity k d / (k + 1)): its time, and frac = that time / the measured
    launch time, defined as the main roofline's (above 1: faster than any mapper without
    source reuse could be)."""
    t_tc = alg["flop"] / (peaks["bf16"] * 1e12)
    t_hbm = alg["no_reuse_bytes_per_token"] * w.n_tokens / (peaks["hbm"] * 1e9)
    ms = 1e3 * max(t_tc, t_hbm)
    return {"bytes_per_token": alg["no_reuse_bytes_per_token"],
            "intensity_flop_per_byte": alg["no_reuse_intensity"], "roofline_ms": ms,
            "bound": "tensor" if t_tc >= t_hbm else "hbm", "frac": ms / ms_step}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sustained=d.get("bf16_tflops_sustained"),
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, source="fallback")


def code_only(text):
    """Source text without // comments and blank lines (a comment edit keeps the hash)."""
    out = []
    for ln in text.splitlines():
        ln = re.sub(r"//.*$", "", ln).rstrip()
        if ln:
            out.append(ln)
    return "\n".join(out)


def kernel_hash(read=None):
    """sha256 (16 hex digits) of the tensor-core kernel's code, the key of the committed
    traffic figure."""
    read = read or (lambda f: open(os.path.join(ROOT, f), encoding="utf-8").read())
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        h.update(code_only(read(f)).encode())
    return h.hexdigest()[:16]


def committed_traffic(w):
    """dram bytes per launch from the committed ncu summary, if taken on this kernel and on
    the named workload as defined (no --override: a changed field such as the weight dtype
    changes the kernel instance or its traffic)."""
    if not os.path.exists(TRAFFIC_FILE) or syn.WORKLOADS.get(w.name) != w:
        return None
    workload = w.name
    kv = {}
    for ln in open(TRAFFIC_FILE):
        if ":" in ln and not ln.startswith("#"):
            a, b = ln.split(":", 1)
            kv[a.strip()] = b.strip()
    if kv.get("kernel_source_sha256_16") != kernel_hash() or kv.get("workload") != workload:
        return None
    try:
        return float(kv["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        rows = []
        for ln in (self.out or "").splitlines():
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append(dict(sm=float(parts[1]), smax=float(parts[2]), power=float(parts[3]),
                                 hw=parts[5], hwt=parts[6], swt=parts[7], pcap=parts[8]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"]}
        loaded = [r for r in rows if r["power"] > 200.0] or rows
        reasons = set()
        for r in loaded:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("pcap", "sw_power_cap")):
                if r[key].lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in loaded),
                "sm_max_mhz": max(r["smax"] for r in rows), "reasons": sorted(reasons),
                "samples": len(rows), "samples_under_load": len(loaded),
                "power_w_max": max(r["power"] for r in rows)}


def measure_link(h_src, h_dst, d_src, d_dst, dev, reps=3):
    """Host link bandwidth of this machine in GB/s, from pinned copies of the step's own
    buffers: host->device alone, device->host alone, and both at once on two streams
    (best of `reps`).  The e2e copy floor of a step follows from these."""
    def timed(fns):
        best = float("inf")
        for _ in range(reps):
            streams = [torch.cuda.Stream(dev) for _ in fns]
            torch.cuda.synchronize(dev)
            t0 = time.perf_counter()
            for s, fn in zip(streams, fns):
                with torch.cuda.stream(s):
                    fn()
            torch.cuda.synchronize(dev)
            best = min(best, time.perf_counter() - t0)
        return best
    hb = h_src.numel() * h_src.element_size()
    db = h_dst.numel() * h_dst.element_size()
    t_h = timed([lambda: d_src.copy_(h_src, non_blocking=True)])
    t_d = timed([lambda: h_dst.copy_(d_dst, non_blocking=True)])
    # both directions at once on equal byte counts, so that neither copy runs alone at the end
    n = min(h_src.numel(), h_dst.numel())
    hs, ds = h_src.view(-1)[:n], d_src.view(-1)[:n]
    hd, dd = h_dst.view(-1)[:n], d_dst.view(-1)[:n]
    t_b = timed([lambda: ds.copy_(hs, non_blocking=True), lambda: hd.copy_(dd, non_blocking=True)])
    nb = n * h_src.element_size()
    return {"h2d_gbs": hb / t_h / 1e9, "d2h_gbs": db / t_d / 1e9, "both_gbs": 2 * nb / t_b / 1e9,
            "measured_on": "pinned copies: one key cache each way alone (%.2f GB in, %.2f GB out), then "
                           "%.2f GB each way at once; best of %d" % (hb / 1e9, db / 1e9, nb / 1e9, reps)}


def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        return rank, world, local, dist
    return 0, 1, 0, None


def barrier(dist):
    if dist is not None:
        dist.barrier()


def max_over_ranks(x, dist, dev):
    if dist is None:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world, tokens_per_step, steps, ms):
    """Whole-job tokens/s: every rank maps tokens_per_step tokens per step (replicas, weak
    scaling), over the slowest rank's elapsed ms."""
    return world * tokens_per_step * steps / (ms / 1e3)


# ------------------------------------------------------------------ oracle leg ----

def _exact_f64(t):
    """Exact float64 values of a CPU tensor of bfloat16 (decoded bit pattern) or float32."""
    from oracle import bf16 as obf16
    if t.dtype == torch.bfloat16:
        return obf16.decode(t.contiguous().view(torch.int16).numpy().view(np.uint16))
    return t.double().numpy()


def _oracle_mode(w):
    """The oracle's rounding model for a workload: the bf16 forward for bf16 caches."""
    return "exact" if w.cache_dtype == "f32" else "bf16fwd"


def oracle_sample_rate(w, budget_s, seed=0, ctx_sel=None):
    """Time the float64 oracle (as it stands) on a bounded sample of the workload's
    tokens.  Returns (tokens/s, tokens, seconds, threads)."""
    from oracle import mapper as omap
    from oracle import selection as osel
    W, b = syn.weights(w)
    Wf, bf = _exact_f64(W), _exact_f64(b)
    sel = osel.select_topk(syn.selection_scores(w), w.k)
    pos = syn.positions(w)
    rng = np.random.default_rng(seed)

    def run(n):
        rows = np.stack([rng.integers(0, w.B, n), rng.integers(0, w.T, n)], axis=1)
        sk = syn.source_rows(w, 0, rows)
        sv = syn.source_rows(w, 1, rows)
        skf, svf = _exact_f64(sk), _exact_f64(sv)
        p = pos[rows[:, 0], rows[:, 1]]
        t0 = time.perf_counter()
        omap.map_tokens(skf, svf, p, sel, Wf, bf, w.theta_s, w.theta_t, mode=_oracle_mode(w), head_mix=w.head_mix,
                        style=w.rope_style)
        return time.perf_counter() - t0

    n, dt = 8, run(8)
    while dt < 0.2 * budget_s and n < w.n_tokens:
        n = min(w.n_tokens, int(n * min(8.0, max(2.0, 0.5 * budget_s / max(dt, 1e-3)))))
        dt = run(n)
    return n / dt, n, dt, blas_threads()


def oracle_one_core(w, budget_s=6.0):
    """The oracle's rate with one BLAS thread: a fresh interpreter (exec, no CUDA) with the
    BLAS thread counts set to 1 runs oracle_sample_rate on the same workload.  Returns
    {"value", "sample"} or None if the child fails."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    fields = json.dumps({k: (list(v) if isinstance(v, tuple) else v) for k, v in dataclasses.asdict(w).items()})
    code = ("import json, sys; sys.path.insert(0, %r); import bench; "
            "from paper_2608_03893_gb300 import synthetic as syn; "
            "d = json.loads(sys.argv[1]); "
            "d = {k: (tuple(v) if isinstance(v, list) else v) for k, v in d.items()}; "
            "r = bench.oracle_sample_rate(syn.Workload(**d), budget_s=%f, seed=1); "
            "print(json.dumps(r))" % (ROOT, budget_s))
    try:
        out = subprocess.run([sys.executable, "-c", code, fields], env=env, capture_output=True, text=True,
                             timeout=120 + 10 * budget_s)
        rate, n, dt, threads = json.loads(out.stdout.strip().splitlines()[-1])
    except Exception:
        return None
    return {"value": rate, "threads": threads, "sample": "%d tokens, %.1f s" % (n, dt)}


def blas_threads():
    try:
        from threadpoolctl import threadpool_info
        info = threadpool_info()
        if info:
            return int(max(i.get("num_threads", 1) for i in info))
    except Exception:
        pass
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS"):
        if os.environ.get(var, "").isdigit():
            return int(os.environ[var])
    return os.cpu_count() or 1


def reference_arm(args, w, config):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from oracle import mapper as omap
    from oracle import selection as osel
    # size one step so that warmup + steps stay within a few minutes
    rate, n_cal, dt_cal, cores = oracle_sample_rate(w, budget_s=2.0)
    per_step = max(1, min(w.n_tokens, int(rate * 150.0 / max(1, args.steps + args.warmup))))
    W, b = syn.weights(w)
    Wf, bf = _exact_f64(W), _exact_f64(b)
    sel = osel.select_topk(syn.selection_scores(w), w.k)
    pos = syn.positions(w)
    # one seeded sample of the workload's tokens, generated once (its generation is not
    # oracle work) and mapped by every step
    rng = np.random.default_rng(7)
    rows = np.stack([rng.integers(0, w.B, per_step), rng.integers(0, w.T, per_step)], axis=1)
    skf, svf = _exact_f64(syn.source_rows(w, 0, rows)), _exact_f64(syn.source_rows(w, 1, rows))
    prow = pos[rows[:, 0], rows[:, 1]]
    times, toks = [], 0
    step_budget = 150.0 / max(1, args.steps + args.warmup)
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        omap.map_tokens(skf, svf, prow, sel, Wf, bf, w.theta_s, w.theta_t,
                        mode=_oracle_mode(w), head_mix=w.head_mix, style=w.rope_style)
        dt = time.perf_counter() - t0
        if i >= args.warmup:
            times.append(dt)
            toks += per_step
        elif dt > 1.2 * step_budget and per_step > 1:
            # the oracle's rate per token falls as the sample grows: the warm-up steps trim
            # the sample to the step's share of the time budget before the timed steps
            per_step = max(1, int(per_step * step_budget / dt))
            skf, svf, prow = skf[:, :, :per_step], svf[:, :, :per_step], prow[:per_step]
    total = sum(times)
    value = toks / total
    sample = "%d random tokens (of %d), the same sample every step, float64 oracle, numpy BLAS" % (per_step, w.n_tokens)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config,
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# -------------------------------------------------------------------- GPU leg -----

def make_mapper(w, dev_index):
    W, b = syn.weights(w)
    cfg, keep = kvx.config_from_tensors(
        src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k, theta_s=w.theta_s,
        theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b, scores=syn.selection_scores(w),
        head_mix=kvx.KVX_CROSS_HEAD if w.head_mix == "cross_head" else kvx.KVX_PER_HEAD,
        rope_style=kvx.KVX_ROPE_INTERLEAVED if w.rope_style == "interleaved" else kvx.KVX_ROPE_HALF)
    return kvx.kvx_create(cfg, dev_index)




def paged_bench(args, w):
    """Multi-turn paged handoff (Sec. 4.5): every sequence's cache lives in one paged pool
    whose block table covers its final length (initial length + turns x T tokens); a step
    maps all turns in order, each turn's new tokens at their absolute positions from that
    turn's own source cache.  One launch per turn.  value = mapped tokens per step / step
    time; the roofline is taken per launch (one turn) on the average launch time."""
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream(dev)
    sp = stream.cuda_stream
    ctx = make_mapper(w, 0)
    kernel_id = kvx.kvx_get_kernel(ctx, paged=True)
    kernel_name = kvx.KERNEL_NAMES[kernel_id]
    L0 = syn.initial_lengths(w)
    table, n_blocks = syn.persistent_block_table(w, L0)
    tbl = torch.from_numpy(table).to(dev)
    pool_k = torch.empty((w.Lt, n_blocks, w.H, w.block_size, w.d), dtype=torch.bfloat16, device=dev)
    pool_v = torch.empty_like(pool_k)
    pool_k.view(torch.int16).fill_(0x7FBF)
    pool_v.view(torch.int16).fill_(0x7FBF)
    tgt = kvx.tgt_paged_from_tensors(pool_k, pool_v, tbl, w.block_size)
    turns = []
    for j in range(w.turns):
        sk = syn.source_cache(w, 0, device=dev, turn=j)
        sv = syn.source_cache(w, 1, device=dev, turn=j)
        pos = torch.from_numpy(syn.positions(w, j, L0)).to(dev)
        turns.append((sk, sv, pos, kvx.src_from_tensors(sk, sv)))

    def step():
        for sk, sv, pos, src in turns:
            kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, sp)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    assert kvx.kvx_get_status(ctx, sp) == kvx.KVX_OK
    steps = max(1, args.steps)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(0) as clk:
        torch.cuda.synchronize()
        ev0.record(stream)
        for _ in range(steps):
            step()
        ev1.record(stream)
        torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1) / steps
    st = kvx.kvx_get_status(ctx, sp)
    tokens = w.n_tokens * w.turns

    # e2e: each turn's source caches and positions copied from pinned host memory inside
    # the timed region (one turn's host buffers, copied into every turn's device buffers),
    # then the map; the mapped target stays in the device pool the target model reads, so
    # the step's device-to-host read is the 4-byte status word
    hk = torch.empty(turns[0][0].shape, dtype=torch.bfloat16, pin_memory=True)
    hv = torch.empty_like(hk, pin_memory=True)
    hk.copy_(turns[0][0])
    hv.copy_(turns[0][1])
    hpos = [torch.from_numpy(syn.positions(w, j, L0)).pin_memory() for j in range(w.turns)]
    h2d = w.turns * (hk.numel() * 2 + hv.numel() * 2 + hpos[0].numel() * 4)

    def e2e_step():
        for (sk, sv, pos, src), hp in zip(turns, hpos):
            sk.copy_(hk, non_blocking=True)
            sv.copy_(hv, non_blocking=True)
            pos.copy_(hp, non_blocking=True)
            kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, sp)
        return kvx.kvx_get_status(ctx, sp)

    e2e_steps = max(1, min(args.e2e_steps or 3, 5))
    e2e_step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(e2e_steps):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    ems = e0.elapsed_time(e1) / e2e_steps
    kvx.kvx_destroy(ctx)

    alg = algorithmic(w)                       # one launch = one turn
    peaks = load_peaks()
    launch_s = ms / w.turns / 1e3
    t_tc = alg["flop"] / (peaks["bf16"] * 1e12)
    t_hbm = alg["bytes"] / (peaks["hbm"] * 1e9)
    bound = "tensor" if t_tc >= t_hbm else "hbm"
    if bound == "tensor":
        achieved, peak, unit = alg["flop"] / launch_s / 1e12, peaks["bf16"], "TFLOP/s"
    else:
        achieved, peak, unit = alg["bytes"] / launch_s / 1e9, peaks["hbm"], "GB/s"
    clocks = clk.summary()
    line = {"metric": METRIC, "value": tokens / (ms / 1e3), "unit": UNIT, "n_gpus": 1, "steps": steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name + " (persistent pool, %d turns per step)" % w.turns,
                       "src_layers": w.Ls, "tgt_layers": w.Lt, "kv_heads": w.H, "head_dim": w.d, "k": w.k,
                       "batch": w.B, "tokens_per_turn": w.T, "turns": w.turns, "tokens_per_step": tokens,
                       "pool_blocks": n_blocks, "pool_gb": 2 * pool_k.numel() * 2 / 1e9,
                       "initial_lengths": [int(x) for x in L0], "layout": "paged (16-token blocks)",
                       "l2": "no flush: each turn streams %.1f GB vs 129 MB L2" % (alg["bytes"] / 1e9)},
            "clocks": clocks, "status": kvx.kvx_status_string(st),
            "kcycles_per_step": ms * clocks["sm_mhz"] if clocks.get("sm_mhz") else None,
            "per_turn_ms": ms / w.turns,
            "e2e": {"value": tokens / (ems / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": 4,
                    "steps": e2e_steps, "ms_per_step": ems,
                    "api": "per turn: pinned-host copies of the source caches and positions + kvx_map into the "
                           "device pool; kvx_get_status read at the end of the step"},
            "gpu_launches": steps * w.turns * (2 if kernel_id == 3 else 1),
            "roofline": {"bound": bound, "achieved": achieved, "peak": peak, "unit": unit, "frac": achieved / peak,
                         "traffic": None, "per": "launch (one turn, %d tokens)" % w.n_tokens,
                         "peak_source": "%s (bf16 burst; HBM copy)" % peaks["source"],
                         "other": {"hbm_frac": alg["bytes"] / launch_s / 1e9 / peaks["hbm"],
                                   "tensor_frac": alg["flop"] / launch_s / 1e12 / peaks["bf16"]},
                         "algorithmic": {"flop_per_launch": alg["flop"], "bytes_per_launch": alg["bytes"]}},
            "cpu_baseline": None, "kernel": kernel_name + ", paged epilogue"}
    print(json.dumps(line), flush=True)
    return 0


# The solve runs in float-float arithmetic on the FP32 lanes: one pair FMA is 15 FP32
# instructions (two_prod by FMA, two_sum, fast_two_sum), and counts as 2 FLOP.
FF_FMA_INSTR = 15
FF_PEAK_TFLOPS = 152 * 128 * 2.07e9 / FF_FMA_INSTR * 2 / 1e12


def fit_bench(args, w):
    """Ridge fit of every (target layer, K|V, head) on N = B*T calibration tokens of the
    workload's shapes.  One step = one kvx_fit_ridge call (mean, Gram and solve kernels,
    synchronous).  Roofline: the Gram blocks' fp32 FFMA work against the FP32 peak derived
    from the unit counts (152 SMs x 128 lanes x 2 x 2070 MHz); the fp64 solve is listed."""
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    sp = torch.cuda.current_stream(dev).cuda_stream
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = torch.from_numpy(syn.positions(w)).to(dev)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    cross = w.head_mix == "cross_head"
    mix = kvx.KVX_CROSS_HEAD if cross else kvx.KVX_PER_HEAD
    F = w.F
    R = w.H * w.d if cross else w.d             # right-hand sides per system
    W = torch.empty((w.Lt, 2, w.H, F, w.d), dtype=torch.float32, device=dev)
    b = torch.empty((w.Lt, 2, w.H, w.d), dtype=torch.float32, device=dev)
    src, tgt = kvx.src_from_tensors(sk, sv), kvx.src_from_tensors(tk, tv)
    # one caller workspace, allocated once (no per-call allocation inside the timed region)
    ws_bytes = kvx.kvx_fit_workspace_bytes(w.Ls, w.Lt, w.H, w.d, w.k, w.theta_s, w.theta_t, 0.01, sel, w.B, w.T,
                                           head_mix=mix)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)

    def step():
        kvx.kvx_fit_ridge(w.Ls, w.Lt, w.H, w.d, w.k, w.theta_s, w.theta_t, 0.01, sel, src, tgt, w.B, w.T,
                          pos.data_ptr(), W.data_ptr(), b.data_ptr(), sp, workspace_ptr=ws.data_ptr(),
                          workspace_bytes=ws_bytes, head_mix=mix)

    for _ in range(args.warmup):
        step()
    steps = max(1, min(args.steps, 20))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    phase = [0.0] * 4
    with ClockSampler(0) as clk:
        torch.cuda.synchronize()
        e0.record()
        for _ in range(steps):
            step()
            phase = [a + b for a, b in zip(phase, kvx.kvx_last_phase_ms())]
        e1.record()
        torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    phase = [p / steps for p in phase]
    n_sys = w.Lt * 2 * (1 if cross else w.H)
    N = w.n_tokens
    # Source-pair blocks XsaᵀXsb depend only on the two source layers, so every distinct
    # pair of the selection is one Gram block per (K|V, head) -- per (K|V, head pair) in
    # cross-head mode, where one layer with itself needs only H(H+1)/2 of them; each target
    # layer adds its cross blocks XᵀY (k per head, or k H H).  A block is N d² fused
    # multiply-adds.
    sel_np = np.asarray(sel).reshape(w.Lt, w.k)
    pairs = {(max(int(a), int(c)), min(int(a), int(c))) for row in sel_np for i, a in enumerate(row) for c in row[:i + 1]}
    blk = 2.0 * N * w.d * w.d
    if cross:
        n_src_blocks = sum(w.H * (w.H + 1) // 2 if a == c else w.H * w.H for a, c in pairs)
        gram_flop = 2 * (n_src_blocks + w.Lt * w.k * w.H * w.H) * blk
        gram_flop_unshared = n_sys * (F // w.d) * (F // w.d + 1) // 2 * blk + 2 * w.Lt * w.k * w.H * w.H * blk
    else:
        gram_flop = 2 * w.H * (len(pairs) + w.Lt * w.k) * blk
        gram_flop_unshared = n_sys * (w.k * (w.k + 1) // 2 + w.k) * blk
    solve_flop = n_sys * (F ** 3 / 3.0 + 2.0 * F * F * R)
    # dominant kernel: the fp64 solve (Cholesky + two triangular solves per system)
    achieved = solve_flop / (phase[3] / 1e3) / 1e12
    # the Gram kernel issues four bf16 MMAs per product (hi/lo split of both operands)
    gram_tc_tflops = 4.0 * gram_flop / (phase[2] / 1e3) / 1e12
    pk = load_peaks()
    line = {"metric": "ridge-fit calibration tokens/s", "value": N / (ms / 1e3), "unit": "tokens/s", "n_gpus": 1,
            "steps": steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16 caches, bf16x2-split tensor-core Gram (fp32 accumulate), float-float solve",
            "data": "synthetic",
            "config": {"workload": w.name + " (fit)", "src_layers": w.Ls, "tgt_layers": w.Lt, "kv_heads": w.H,
                       "head_dim": w.d, "k": w.k, "calibration_tokens": N, "systems": n_sys, "lambda": 0.01,
                       "head_mix": w.head_mix, "features": F, "rhs_per_system": R,
                       "workspace_gb": ws_bytes / 1e9},
            "clocks": clk.summary(),
            "gpu_launches": 4 * steps,
            "phase_ms": {"column_sums": phase[0], "pack": phase[1], "gram_tc": phase[2], "solve": phase[3]},
            "roofline": {"bound": "alu", "achieved": achieved, "peak": FF_PEAK_TFLOPS, "unit": "TFLOP/s",
                         "frac": achieved / FF_PEAK_TFLOPS, "traffic": None,
                         "kernel": ("fit_solve_xh_kernel" if cross else "fit_solve_kernel") + " (float-float on the FP32 lanes)",
                         "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2070 MHz / 15 FP32 instructions per "
                                        "float-float FMA x 2 FLOP (the FP64-equivalent work; GB300's FP64 "
                                        "units give 1.25 TFLOP/s nominal)",
                         "algorithmic": {"solve_fp64_flop_per_step": solve_flop, "gram_flop_per_step": gram_flop,
                                         "gram_blocks_source_pairs": len(pairs),
                                         "gram_flop_without_pair_sharing": gram_flop_unshared},
                         "other": {"gram_tc_kernel": {"bound": "tensor", "achieved": gram_tc_tflops,
                                                      "peak": pk["bf16"], "frac": gram_tc_tflops / pk["bf16"],
                                                      "unit": "TFLOP/s (bf16 MMA, four per product)"}}},
            "kernel": "gram_pack_kernel<0> + gram_pack_kernel<1> + gram_tc_kernel + "
                      + ("fit_solve_xh_kernel" if cross else "fit_solve_kernel")}
    print(json.dumps(line), flush=True)
    return 0


def probe_bench(args, w):
    """Single-source R^2 probe (kvx_r2_probe) of every (target layer, source layer) pair on
    N = B*T calibration tokens of the workload's shapes.  One step = one kvx_r2_probe call
    (column sums, pack, tensor-core Gram blocks, factor / score / reduce kernels,
    synchronous).  Roofline: the tensor-core Gram kernel (four bf16 MMAs per product) against
    the measured bf16 peak."""
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    sp = torch.cuda.current_stream(dev).cuda_stream
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = torch.from_numpy(syn.positions(w)).to(dev)
    scores = torch.empty((w.Lt, w.Ls), dtype=torch.float64, device=dev)
    src, tgt = kvx.src_from_tensors(sk, sv), kvx.src_from_tensors(tk, tv)
    ws_bytes = kvx.kvx_r2_probe_workspace_bytes(w.Ls, w.Lt, w.H, w.d, w.theta_s, w.theta_t, w.B, w.T)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)

    def step():
        kvx.kvx_r2_probe(w.Ls, w.Lt, w.H, w.d, w.theta_s, w.theta_t, src, tgt, w.B, w.T, pos.data_ptr(),
                         scores.data_ptr(), None, sp, workspace_ptr=ws.data_ptr(), workspace_bytes=ws_bytes)

    for _ in range(args.warmup):
        step()
    steps = max(1, min(args.steps, 20))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    phase = [0.0] * 4
    with ClockSampler(0) as clk:
        torch.cuda.synchronize()
        e0.record()
        for _ in range(steps):
            step()
            phase = [a + b for a, b in zip(phase, kvx.kvx_last_phase_ms())]
        e1.record()
        torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    phase = [p / steps for p in phase]
    N = w.n_tokens
    blocks = 2 * w.H * w.Ls * (w.Lt + 1)              # C blocks of every pair + A of every source
    gram_flop = blocks * 2.0 * N * w.d * w.d          # algorithmic: one product per token and entry pair
    achieved = 4.0 * gram_flop / (phase[2] / 1e3) / 1e12
    pk = load_peaks()
    line = {"metric": "R2-probe calibration tokens/s", "value": N / (ms / 1e3), "unit": "tokens/s", "n_gpus": 1,
            "steps": steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16 caches, bf16x2-split tensor-core Gram (fp32 accumulate), fp64 Cholesky, fp32 scores",
            "data": "synthetic",
            "config": {"workload": w.name + " (R2 probe)", "src_layers": w.Ls, "tgt_layers": w.Lt, "kv_heads": w.H,
                       "head_dim": w.d, "calibration_tokens": N, "layer_pairs": w.Lt * w.Ls,
                       "workspace_gb": ws_bytes / 1e9},
            "clocks": clk.summary(),
            "gpu_launches": 7 * steps,
            "phase_ms": {"column_sums": phase[0], "pack": phase[1], "gram_tc": phase[2], "factor_score": phase[3]},
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": pk["bf16"], "unit": "TFLOP/s",
                         "frac": achieved / pk["bf16"], "traffic": None, "kernel": "gram_tc_kernel",
                         "peak_source": pk["source"] + " bf16 (four bf16 MMAs per product counted)",
                         "algorithmic": {"gram_blocks": blocks, "gram_flop_per_step": gram_flop}},
            "kernel": "gram_pack_kernel<0> + gram_pack_kernel<1> + gram_tc_kernel + probe kernels"}
    print(json.dumps(line), flush=True)
    return 0


MLP_HIDDEN = 1024   # the paper's MLP baseline width
E2E_CHUNK = 2048    # tokens per chunk of the host-buffer pipeline (best of 1024..16384 in three sweeps)


def mlp_bench(args, w):
    """MLP mapper apply (kvx_mlp_map): the three-layer ReLU MLP per (target layer, K|V, head)
    on the cross-head source feature, synthetic seeded weights on the device.  One step =
    one kvx_mlp_map call (key strip + three GEMM passes, synchronous) with a caller
    workspace.  Roofline: tensor-bound, the GEMM FLOPs against the measured bf16 peak."""
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    sp = torch.cuda.current_stream(dev).cuda_stream
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    pos = torch.from_numpy(syn.positions(w)).to(dev)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    hid, ds = MLP_HIDDEN, w.k * w.H * w.d
    g = torch.Generator(device=dev).manual_seed(w.seed + 77)
    shape = (w.Lt, 2, w.H)
    P = dict(W1=torch.randn(*shape, hid, ds, generator=g, device=dev, dtype=torch.bfloat16).mul_(ds ** -0.5),
             b1=torch.randn(*shape, hid, generator=g, device=dev).mul_(0.1),
             W2=torch.randn(*shape, hid, hid, generator=g, device=dev, dtype=torch.bfloat16).mul_((2.0 / hid) ** 0.5),
             b2=torch.randn(*shape, hid, generator=g, device=dev).mul_(0.1),
             W3=torch.randn(*shape, w.d, hid, generator=g, device=dev, dtype=torch.bfloat16).mul_((2.0 / hid) ** 0.5),
             b3=torch.randn(*shape, w.d, generator=g, device=dev).mul_(0.1))
    tk = torch.empty((w.Lt, w.B, w.H, w.T, w.d), dtype=torch.bfloat16, device=dev)
    tv = torch.empty_like(tk)
    cfg = kvx.mlp_config(w.Ls, w.Lt, w.H, w.d, w.k, hid, w.theta_s, w.theta_t, sel,
                         *(P[n].data_ptr() for n in ("W1", "b1", "W2", "b2", "W3", "b3")))
    ws_bytes = kvx.kvx_mlp_workspace_bytes(cfg, w.B, w.T)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    cfg.workspace, cfg.workspace_bytes = ws.data_ptr(), ws_bytes
    src, tgt = kvx.src_from_tensors(sk, sv), kvx.tgt_from_tensors(tk, tv)

    def step():
        kvx.kvx_mlp_map(cfg, src, w.B, w.T, pos.data_ptr(), tgt, sp)

    for _ in range(args.warmup):
        step()
    steps = max(1, min(args.steps, 10))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(0) as clk:
        torch.cuda.synchronize()
        e0.record()
        for _ in range(steps):
            step()
        e1.record()
        torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    N = w.n_tokens
    n_sys = w.Lt * 2 * w.H
    flop = n_sys * N * 2.0 * (ds * hid + hid * hid + hid * w.d)
    achieved = flop / (ms / 1e3) / 1e12
    pk = load_peaks()
    line = {"metric": "MLP-mapper tokens/s", "value": N / (ms / 1e3), "unit": "tokens/s", "n_gpus": 1,
            "steps": steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16 (fp32 accumulate)", "data": "synthetic",
            "config": {"workload": w.name + " (MLP mapper)", "src_layers": w.Ls, "tgt_layers": w.Lt,
                       "kv_heads": w.H, "head_dim": w.d, "k": w.k, "hidden": hid, "d_s": ds, "batch": w.B,
                       "seq_len": w.T, "weights_gb": sum(t.numel() * t.element_size() for t in P.values()) / 1e9,
                       "workspace_gb": ws_bytes / 1e9,
                       "l2": "no flush: each step reads %.1f GB of weights vs 129 MB L2" % (
                           sum(t.numel() * t.element_size() for t in P.values()) / 1e9)},
            "clocks": clk.summary(),
            "gpu_launches": 4 * steps,
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": pk["bf16"], "unit": "TFLOP/s",
                         "frac": achieved / pk["bf16"], "traffic": None, "kernel": "tc_mlp_kernel (3 passes) + strip",
                         "peak_source": pk["source"] + " bf16 burst",
                         "algorithmic": {"flop_per_step": flop, "flop_per_token": flop / N}},
            "kernel": "xh_strip_kernel + tc_mlp_kernel x 3"}
    print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="kvx", choices=["kvx", "reference"])
    ap.add_argument("--workload", default=syn.HEADLINE)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=None)
    ap.add_argument("--fit", action="store_true",
                    help="time the ridge fit (kvx_fit_ridge) on the workload's shapes instead of the map")
    ap.add_argument("--override", default="",
                    help="comma-separated workload fields for a smaller case of the same kernel, e.g. "
                         "Lt=16,T=4096 (profiling captures)")
    ap.add_argument("--mlp", action="store_true",
                    help="time the MLP mapper apply (kvx_mlp_map, hidden 1024) on the workload's shapes")
    ap.add_argument("--probe", action="store_true",
                    help="time the single-source R^2 probe (kvx_r2_probe) on the workload's shapes")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    over = {}
    for kv in filter(None, args.override.split(",")):
        key, val = kv.split("=")
        over[key.strip()] = type(getattr(syn.WORKLOADS[args.workload], key.strip()))(val)
    w = syn.workload(args.workload, **over)
    if args.fit:
        return fit_bench(args, w)
    if args.probe:
        return probe_bench(args, w)
    if args.mlp:
        return mlp_bench(args, w)
    if w.paged and args.impl != "reference":
        return paged_bench(args, w)
    alg = algorithmic(w)
    config = {"workload": w.name, "src_layers": w.Ls, "tgt_layers": w.Lt, "kv_heads": w.H,
              "head_dim": w.d, "k": w.k, "batch": w.B, "seq_len": w.T, "tokens_per_step": w.n_tokens,
              "rope_theta": w.theta_t, "layout": "paged" if w.paged else "contiguous",
              "parallelism": "replicas x%d" % args.gpus,
              "l2": "no flush: each step streams %.1f GB (source read + target write) vs 129 MB L2"
                    % (alg["bytes"] / 1e9)}
    if w.rope_style != "half":
        config["rope_pairs"] = w.rope_style
    if args.impl == "reference":
        return reference_arm(args, w, config)

    rank, world, local, dist = dist_setup(args.gpus)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    sp = stream.cuda_stream

    ctx = make_mapper(w, local)
    kernel_id = kvx.kvx_get_kernel(ctx)
    sk = syn.source_cache(w, 0, device=dev)
    sv = syn.source_cache(w, 1, device=dev)
    pos_np = syn.positions(w)
    pos = torch.from_numpy(pos_np).to(dev)
    tk = torch.empty((w.Lt, w.B, w.H, w.T, w.d), dtype=torch.bfloat16, device=dev)
    tv = torch.empty_like(tk)
    src, tgt = kvx.src_from_tensors(sk, sv), kvx.tgt_from_tensors(tk, tv)

    def step():
        kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, sp)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    assert kvx.kvx_get_status(ctx, sp) == kvx.KVX_OK
    assert not torch.isnan(tk).any().item()

    # one event between consecutive launches: the total and each launch's own time
    evs_k = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    with ClockSampler(local) as clk:
        barrier(dist)
        torch.cuda.synchronize()
        evs_k[0].record(stream)
        for i in range(args.steps):
            step()
            evs_k[i + 1].record(stream)
        torch.cuda.synchronize()
        barrier(dist)
    ms = evs_k[0].elapsed_time(evs_k[-1])
    per_launch = [evs_k[i].elapsed_time(evs_k[i + 1]) for i in range(args.steps)]
    ms = max_over_ranks(ms, dist, dev)
    st = kvx.kvx_get_status(ctx, sp)
    ms_step = ms / args.steps
    value = job_rate(world, w.n_tokens, args.steps, ms)

    # ---- e2e: host buffers through the C ABI, copies inside the timed region
    e2e_steps = args.e2e_steps or max(3, min(args.steps, 40))
    hk = torch.empty(sk.shape, dtype=sk.dtype, pin_memory=True)
    hv = torch.empty(sv.shape, dtype=sv.dtype, pin_memory=True)
    hk.copy_(sk)
    hv.copy_(sv)
    hpos = torch.from_numpy(pos_np).pin_memory()
    ok_ = torch.empty(tk.shape, dtype=tk.dtype, pin_memory=True)
    ov_ = torch.empty(tv.shape, dtype=tv.dtype, pin_memory=True)
    h2d = hk.numel() * 2 + hv.numel() * 2 + hpos.numel() * 4
    d2h = ok_.numel() * 2 + ov_.numel() * 2

    # contiguous targets: the public host-buffer call (kvx_map_host), which overlaps the
    # copies of one chunk of tokens with the map of the next; paged targets: copies around
    # kvx_map on the stream
    pipe = None
    if not w.paged:
        chunk = E2E_CHUNK if w.T > E2E_CHUNK else w.T
        pipe = kvx.kvx_host_pipe_create(ctx, w.B, chunk)
        h_src, h_tgt = kvx.src_from_tensors(hk, hv), kvx.tgt_from_tensors(ok_, ov_)

    def e2e_step():
        if pipe is not None:
            kvx.kvx_map_host(pipe, h_src, w.T, hpos.data_ptr(), h_tgt, sp)
            return
        sk.copy_(hk, non_blocking=True)
        sv.copy_(hv, non_blocking=True)
        pos.copy_(hpos, non_blocking=True)
        kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, sp)
        ok_.copy_(tk, non_blocking=True)
        ov_.copy_(tv, non_blocking=True)

    for _ in range(3):
        e2e_step()
    torch.cuda.synchronize()
    barrier(dist)
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(e2e_steps + 1)]
    evs[0].record(stream)
    for i in range(e2e_steps):
        e2e_step()
        evs[i + 1].record(stream)
    torch.cuda.synchronize()
    barrier(dist)
    per_step = [evs[i].elapsed_time(evs[i + 1]) for i in range(e2e_steps)]
    ems = max_over_ranks(evs[0].elapsed_time(evs[-1]), dist, dev)
    e2e_value = job_rate(world, w.n_tokens, e2e_steps, ems)
    link = measure_link(hk, ok_, sk, tk, dev)
    floor_ms = max(h2d / link["h2d_gbs"], d2h / link["d2h_gbs"], (h2d + d2h) / link["both_gbs"]) / 1e6
    e2e_api = "kvx_map_host (chunks of %d tokens)" % chunk if pipe is not None else "copies + kvx_map"
    if pipe is not None:
        kvx.kvx_host_pipe_destroy(pipe)
    del hk, hv, ok_, ov_

    kvx.kvx_destroy(ctx)
    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0

    peaks = load_peaks()
    t_tc = alg["flop"] / (peaks["bf16"] * 1e12)
    t_hbm = alg["bytes"] / (peaks["hbm"] * 1e9)
    launch_s = ms_step / 1e3                  # one launch per step
    bound = "tensor" if t_tc >= t_hbm else "hbm"
    if bound == "tensor":
        achieved, peak, unit = alg["flop"] / launch_s / 1e12, peaks["bf16"], "TFLOP/s"
    else:
        achieved, peak, unit = alg["bytes"] / launch_s / 1e9, peaks["hbm"], "GB/s"
    roofline = {"bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
                "frac": achieved / peak, "traffic": committed_traffic(w),
                "peak_source": "%s (bf16 burst; HBM copy)" % peaks["source"],
                "roofline_ms": 1e3 * max(t_tc, t_hbm),
                "other": {"hbm_achieved_gbs": alg["bytes"] / launch_s / 1e9, "hbm_peak_gbs": peaks["hbm"],
                          "hbm_frac": alg["bytes"] / launch_s / 1e9 / peaks["hbm"],
                          "tensor_achieved_tflops": alg["flop"] / launch_s / 1e12,
                          "tensor_frac": alg["flop"] / launch_s / 1e12 / peaks["bf16"],
                          # against cuBLAS run back to back under the power cap (the
                          # regime a long bench run settles in); context, not the headline
                          "tensor_frac_of_sustained": (alg["flop"] / launch_s / 1e12 / peaks["bf16_sustained"]
                                                       if peaks.get("bf16_sustained") else None),
                          "no_reuse": no_reuse_bound(alg, w, peaks, ms_step)},
                "algorithmic": {"flop_per_launch": alg["flop"], "bytes_per_launch": alg["bytes"],
                                "flop_per_token": alg["flop_per_token"],
                                "bytes_per_token": alg["bytes_per_token"],
                                "weight_bytes": alg["weight_bytes"]}}
    cpu = None
    if not args.no_cpu_baseline:
        rate, n, dt, cores = oracle_sample_rate(w, budget_s=12.0)
        cpu = {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": "%d random tokens of the workload (all %d layers x %d heads x K,V), "
                         "float64 numpy oracle, %.1f s" % (n, w.Lt, w.H, dt)}
        cpu["one_core"] = oracle_one_core(w)
    clocks = clk.summary()
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": config,
            "clocks": clocks, "status": kvx.kvx_status_string(st),
            # ms per step x median SM MHz = thousands of SM cycles per step: compares runs
            # taken at different clocks (a power-capped long run against a short burst)
            "kcycles_per_step": (ms_step * clocks["sm_mhz"] if clocks.get("sm_mhz") else None),
            "ms_per_step_median": statistics.median(per_launch), "ms_per_step_min": min(per_launch),
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "steps": e2e_steps, "ms_per_step": ems / e2e_steps, "api": e2e_api,
                    "ms_per_step_min": min(per_step), "ms_per_step_median": statistics.median(per_step),
                    "ms_per_step_max": max(per_step),
                    # steps over 1.5 x the median: (index, ms)
                    "slow_steps": [(i, round(x, 1)) for i, x in enumerate(per_step)
                                   if x > 1.5 * statistics.median(per_step)],
                    "link_gbs": link, "copy_floor_ms": floor_ms,
                    "frac_of_copy_floor": floor_ms / (ems / e2e_steps)},
            # one launch per step, or a key-strip launch and the GEMMs on the cross-head kernel
            "gpu_launches": args.steps * (2 if kernel_id == 3 else 1), "roofline": roofline,
            "cpu_baseline": cpu,
            "kernel": kvx.KERNEL_NAMES[kernel_id]}
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
