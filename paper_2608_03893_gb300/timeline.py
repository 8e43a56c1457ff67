"""Per-role timeline of the per-head tensor-core map kernel (profiling utility).

Builds a separate copy of libkvx in a temporary directory whose tc_map_kernel records
clock64 stamps at the start and end of every wait of the first cluster's roles (lane 0
of the MMA issuers, of two epilogue warps and of one prologue warp, both CTAs), maps a
workload a few times with it, and prints where each role's cycles go.  The library the
package ships is not touched and the stamps are not in it.

    python -m paper_2608_03893_gb300.timeline qwen3_14b_32b_t32768_k4 [more workloads]

Needs a GPU and nvcc; the instrumented launch runs a few percent slower than the shipped
kernel.
"""
import collections
import ctypes
import glob
import os
import re
import shutil
import subprocess
import sys
import tempfile

import numpy as np

from . import build as kbuild

ROLES = {0: "issuer, even layers (warp 1)", 5: "issuer, odd layers (warp 3)", 1: "epilogue (warp 4)",
         2: "epilogue (warp 11)", 6: "prologue (warp 12)"}
N_ROLES, N_CTAS, LEN = 7, 2, 1 << 16

# (anchor text in kvx_tc.cu, event name, insert after the anchor?)
PROBES = [
    ("          if (acc_n >= 1 && !wait_bar(smem_u32(&acce[iss])", "I_ACCE_W", False),
    ("          tc_fence_after();\n          for (int j = 0; ok && j < k; ++j) {", "I_ACCE_D", False),
    ("              if (!wait_bar(smem_u32(&tready[s * kIssuers + iss])", "I_TREADY_W", False),
    ("              ready_par ^= 1u << s;\n", "I_TREADY_D", True),
    ("              if (!wait_bar(smem_u32(&wfull[st0])", "I_WFULL_W", False),
    ("              const uint32_t b0 = smem_u32(wst + static_cast<size_t>(st0) * kWStageBytes);", "I_WFULL_D", False),
    ("              issued = true;\n", "I_ISSUED", True),
    ("          const bool w_ok = wait_bar(smem_u32(&bias_full[bslot])", "E_BIAS_W", False),
    ("          const bool w_ok = wait_bar(smem_u32(&accf[buf])", "E_ACCF_W", False),
    ("        tc_fence_after();\n        // this warp's staging buffer for the layer", "E_ACCF_D", False),
    ("        __syncwarp();\n        if (lane == 0) mbar_arrive(smem_u32(&bias_empty[bslot]));", "E_COMPUTED", False),
    ("            bulk_commit_group();\n          }\n        }\n", "E_STORED", True),
    ("        bool w_ok =\n            wait_bar(smem_u32(&land_full[lb])", "P_LAND_W", False),
    ("        if ((tl_loaded >> s) & 1u) {\n#pragma unroll\n          for (int i = 0; i < kIssuers; ++i) {", "P_LAND_D", False),
    ("        tc_fence_after();\n        tl_loaded |= 1u << s;", "P_TFREE_D", False),
    ("        tmem_wait_st();\n        tc_fence_before();\n        __syncwarp();\n        if (lane == 0) {", "P_STORED",
     False),
]

# (from event, to event, what the interval is)
SPANS = [
    ("I_ACCE_W", "I_ACCE_D", "wait: accumulator drained by the epilogue"),
    ("I_TREADY_W", "I_TREADY_D", "wait: new source tile in TMEM"),
    ("I_WFULL_W", "I_WFULL_D", "wait: W stage landed"),
    ("I_WFULL_D", "I_ISSUED", "issue 8 pair MMAs"),
    ("E_BIAS_W", "E_ACCF_W", "wait: bias row"),
    ("E_ACCF_W", "E_ACCF_D", "wait: accumulator ready"),
    ("E_ACCF_D", "E_COMPUTED", "TMEM loads, bias, RoPE, bf16, staging"),
    ("E_COMPUTED", "E_STORED", "fence and TMA store"),
    ("P_LAND_W", "P_LAND_D", "wait: source tile landed"),
    ("P_LAND_D", "P_TFREE_D", "wait: TMEM slot released"),
    ("P_TFREE_D", "P_STORED", "strip and TMEM stores"),
]


def _anchor_re(text):
    """A probe's anchor as a pattern that starts at a line start and ignores each line's
    indentation (group 1: the first line's), so re-indenting the kernel keeps it valid."""
    lines = text.split("\n")
    rest = [(" *" + re.escape(ln.lstrip(" "))) if ln else "" for ln in lines[1:]]
    return re.compile(r"(?m)^( *)" + "\n".join([re.escape(lines[0].lstrip(" "))] + rest))


def instrument(src_dir):
    """Write the instrumented kvx_tc.cu into src_dir; returns the event table."""
    path = os.path.join(src_dir, "kvx_tc.cu")
    s = open(path).read()
    events = {}
    head = ("namespace kvx {\n"
            "__device__ unsigned long long g_trace[%d][%d][%d];\n"
            "__device__ unsigned int g_trace_n[%d][%d];\n"
            "namespace {\n\nusing namespace ptx;\n"
            "#define TR(ev) do { if (tr_role >= 0) { if (tr_i < %d) g_trace[tr_cta][tr_role][tr_i] = "
            "(static_cast<unsigned long long>(clock64()) << 8) | (ev); ++tr_i; } } while (0)\n"
            % (N_CTAS, N_ROLES, LEN, N_CTAS, N_ROLES, LEN))
    anchor = "namespace kvx {\nnamespace {\n\nusing namespace ptx;"
    assert s.count(anchor) == 1, "kernel source changed: update the timeline anchors"
    s = s.replace(anchor, head, 1)
    anchor = "  const int warp = threadIdx.x >> 5;\n  const int lane = threadIdx.x & 31;\n"
    assert s.count(anchor) == 1
    s = s.replace(anchor, anchor + (
        "  const int tr_cta = blockIdx.x < 2 ? static_cast<int>(blockIdx.x) : -1;\n"
        "  int tr_role = -1;\n"
        "  if (tr_cta >= 0 && lane == 0) {\n"
        "    if (warp == 1) tr_role = 0; else if (warp == 4) tr_role = 1; else if (warp == 11) tr_role = 2;\n"
        "    else if (warp == 0) tr_role = 3; else if (warp == 2) tr_role = 4; else if (warp == 3) tr_role = 5;\n"
        "    else if (warp == 12) tr_role = 6;\n"
        "  }\n"
        "  unsigned int tr_i = 0;\n"), 1)
    for text, name, after in PROBES:
        found = list(_anchor_re(text).finditer(s))
        assert len(found) == 1, "kernel source changed: probe %s no longer matches" % name
        m = found[0]
        ev = events.setdefault(name, len(events) + 1)
        stamp = "%sTR(%d);\n" % (m.group(1), ev)
        at = m.end() if after else m.start()
        s = s[:at] + stamp + s[at:]
    anchor = "  tc_fence_before();\n  __syncthreads();\n  cluster_sync();   // no arrival or MMA of either CTA still targets the other"
    assert s.count(anchor) == 1
    s = s.replace(anchor, "  if (tr_role >= 0) g_trace_n[tr_cta][tr_role] = tr_i < %d ? tr_i : %d;\n" % (LEN, LEN) + anchor, 1)
    s += ('\nextern "C" __attribute__((visibility("default"))) int kvx_trace_read(unsigned long long* out, '
          'unsigned int* n) {\n  int e = (int)cudaMemcpyFromSymbol(out, kvx::g_trace, sizeof(kvx::g_trace));\n'
          '  return e ? e : (int)cudaMemcpyFromSymbol(n, kvx::g_trace_n, sizeof(kvx::g_trace_n));\n}\n')
    open(path, "w").write(s)
    return events


def build_instrumented(work):
    csrc = os.path.join(work, "pkg", "csrc")
    os.makedirs(csrc)
    shutil.copytree(os.path.join(kbuild.ROOT, "include"), os.path.join(work, "include"))   # ../../include from csrc
    for f in glob.glob(os.path.join(kbuild.CSRC, "*")):
        shutil.copy(f, csrc)
    events = instrument(csrc)
    objs = []
    procs = []
    for f in sorted(glob.glob(os.path.join(csrc, "*.cu")) + glob.glob(os.path.join(csrc, "*.cpp"))):
        o = f + ".o"
        objs.append(o)
        procs.append(subprocess.Popen([kbuild.nvcc()] + kbuild.ARCH + kbuild.COMMON + ["-c", f, "-o", o]))
    if any(p.wait() != 0 for p in procs):
        raise RuntimeError("building the instrumented library failed")
    lib = os.path.join(work, "libkvx_timeline.so")
    subprocess.check_call([kbuild.nvcc()] + kbuild.ARCH + ["-shared", "-o", lib] + objs +
                          ["-lcudart_static", "-ldl", "-lrt", "-lpthread"])
    return lib, events


def summarize(buf, n, events, name, ms):
    inv = {v: k for k, v in events.items()}
    lines = ["## %s (instrumented launch %.3f ms)" % (name, ms), ""]
    t0 = min(int(buf[c, r, 0] >> 8) for c in range(N_CTAS) for r in range(N_ROLES) if n[c, r] > 0)
    for c in range(N_CTAS):
        for r in sorted(ROLES):
            m = int(n[c, r])
            if m == 0:
                continue
            t = (buf[c, r, :m] >> 8).astype(np.int64) - t0
            e = (buf[c, r, :m] & 255).astype(np.int64)
            span = int(t[-1] - t[0])
            acc, cnt, last = collections.Counter(), collections.Counter(), {}
            for ti, ei in zip(t, e):
                ev = inv.get(int(ei))
                for a, b, _ in SPANS:
                    if ev == b and a in last:
                        acc[(a, b)] += ti - last[a]
                        cnt[(a, b)] += 1
                last[ev] = ti
            lines.append("CTA %d, %s: %.2f M cycles" % (c, ROLES[r], span / 1e6))
            for a, b, what in SPANS:
                if cnt[(a, b)]:
                    lines.append("  %-40s %5.1f %%  (%d intervals, mean %d cycles)" % (
                        what, 100.0 * acc[(a, b)] / span, cnt[(a, b)], acc[(a, b)] // cnt[(a, b)]))
            if r in (0, 5):
                issued = int(np.sum(e == events["I_ISSUED"]))
                lines.append("  %-40s %5.1f %%  (%d stages x 8 MMAs x 64 cycles)" % (
                    "tensor work of this issuer", 100.0 * issued * 512 / span, issued))
    return "\n".join(lines)


def main(argv):
    import torch
    from . import kvx
    from . import synthetic as syn
    names = argv or [syn.HEADLINE]
    with tempfile.TemporaryDirectory() as work:
        lib, events = build_instrumented(work)
        kvx.LIB_PATH = lib
        L = kvx.lib()
        L.kvx_trace_read.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
        dev = torch.device("cuda:0")
        for name in names:
            w = syn.workload(name)
            W, b = syn.weights(w)
            cfg, keep = kvx.config_from_tensors(
                src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k, theta_s=w.theta_s,
                theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b, scores=syn.selection_scores(w))
            ctx = kvx.kvx_create(cfg, 0)
            kvx.kvx_set_kernel(ctx, kvx.KVX_KERNEL_TCGEN05)
            sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
            pos = torch.from_numpy(syn.positions(w)).to(dev)
            tk = torch.empty((w.Lt, w.B, w.H, w.T, w.d), dtype=torch.bfloat16, device=dev)
            tv = torch.empty_like(tk)
            src, tgt = kvx.src_from_tensors(sk, sv), kvx.tgt_from_tensors(tk, tv)
            s = torch.cuda.current_stream().cuda_stream
            for _ in range(4):
                kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, s)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, s)
            e1.record()
            torch.cuda.synchronize()
            if kvx.kvx_get_status(ctx, s) != kvx.KVX_OK:
                raise RuntimeError("instrumented launch reported a device error")
            buf = np.zeros((N_CTAS, N_ROLES, LEN), dtype=np.uint64)
            n = np.zeros((N_CTAS, N_ROLES), dtype=np.uint32)
            if L.kvx_trace_read(buf.ctypes.data, n.ctypes.data) != 0:
                raise RuntimeError("reading the timeline failed")
            print(summarize(buf, n, events, name, e0.elapsed_time(e1)), flush=True)
            kvx.kvx_destroy(ctx)
            del sk, sv, tk, tv
            torch.cuda.empty_cache()
    return 0


if __name__ == "__main__":
    sys.exit(main(sys.argv[1:]))
