"""Mutation audit of libkvx's host-side logic against the CPU tests (run by hand, not
collected by pytest; nvcc needed, no GPU).

The audited functions are the ones the CPU tests can reach without a device: the top-k
selection, the mapper-size formula, the RoPE-scaling check, kvx_create's host checks and
selection table, the per-head kernel's load-schedule builder with its entry point, and
the host checks of the fit, probe, MLP and no-alloc entry points (each up to its first
CUDA call).  Each mutant changes
one operator on one code line of one of them (a comparison, a logical operator, a sign,
an index, a constant, a bit of a schedule word) in a private copy of the package; the
copy's build() recompiles that translation unit and relinks, and the CPU tests of the
C ABI run against it.  A mutant that does not build counts as rejected.  Survivors
listed in EQUIVALENT behave the same at the ABI (the same statuses, or a different but
equally valid and optimal schedule), for the reason given; any other survivor is a gap
and makes the audit exit with status 1.

    python tests/host_mutation_audit.py [--jobs 8]      # about 10 minutes on 8 cores

Copies go under ``_build/host_mutation_audit/`` (git-ignored) and are removed afterwards.
"""
import argparse
import concurrent.futures as cf
import os
import re
import shutil
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = "paper_2608_03893_gb300"
TESTS = ["tests/test_abi_cpu.py", "tests/test_schedule_cpu.py", "tests/test_abi_validation_cpu.py",
         "tests/test_abi_bounds_cpu.py"]

# (file, regex of the function's first line, text of the first line that reaches the
# device or None); a function ends at the next "}" in column 0, or before that text
FUNCTIONS = [
    ("kvx_host.cpp", r"^static void topk_rows\(", None),
    ("kvx_host.cpp", r"^const char\* check_rope_scaling\(", None),
    ("kvx_host.cpp", r"^int64_t kvx_mapper_params\(", None),
    ("kvx_host.cpp", r"^kvx_status kvx_select_topk\(", None),
    ("kvx_host.cpp", r"^kvx_status kvx_create\(", "DeviceGuard guard(device);"),
    ("kvx_tc.cu", r"^void build_plan\(", None),
    ("kvx_tc.cu", r"^uint32_t use_bits\(", None),
    ("kvx_tc.cu", r"^KVX_API kvx_status kvx_tc_load_schedule\(", None),
    ("kvx_fit.cu", r"^const char\* check_fit_config\(", None),
    ("kvx_fit.cu", r"^KVX_API kvx_status kvx_fit_ridge\(", "const int sms = sm_count_or_zero();"),
    ("kvx_probe.cu", r"^const char\* check_probe_config\(", None),
    ("kvx_probe.cu", r"^KVX_API kvx_status kvx_r2_probe\(", "cudaStream_t st = static_cast<cudaStream_t>(stream);"),
    ("kvx_mlp.cu", r"^const char\* check_mlp_config\(", None),
    ("kvx_mlp.cu", r"^KVX_API kvx_status kvx_mlp_map\(", "cudaStream_t st = static_cast<cudaStream_t>(stream);"),
    ("kvx_noalloc.cu", r"^extern \"C\" KVX_API kvx_status kvx_map_noalloc\(", "cudaError_t e = cudaGetDevice(&prev);"),
]
# Not audited here: the checks of kvx_map and of the host pipe that follow their NULL-context
# check need a context, and a context needs a GPU (the GPU tests exercise them).

OPS = [
    (r" \+ ", " - "), (r" - ", " + "), (r" < ", " <= "), (r" > ", " >= "), (r" <= ", " < "), (r" >= ", " > "),
    (r" == ", " != "), (r" != ", " == "), (r" && ", " || "), (r" \|\| ", " && "), (r"\bINT_MAX\b", "0"),
    (r"<< i\b", "<< 0"), (r"\|= 4\b", "|= 1"), (r"\|= 1\b", "|= 4"), (r"\b16 <<", "4 <<"), (r"\b4 <<", "16 <<"),
    (r"\bbreak;", ""), (r"\b-1\b", "0"), (r"\+\+i\b", "i += 2"), (r"\bk\b", "1"), (r"\bs\b", "0"),
    (r"\biss\b", "0"), (r"return a < b;", "return a > b;"), (r"return row\[a\] > row\[b\];", "return row[a] < row[b];"),
    (r"std::sort\(idx", "(void)(idx"), (r"\* kIssuers \+ i\]", "* kIssuers]"), (r"\+ 1\b", ""),
]

# (file, mutated line, why the ABI behaves the same).  A mutated line ending in "..." matches
# any line that starts with the text before it.  Text inside string literals (error
# messages) is not mutated.
EQUIVALENT = [
    ("kvx_host.cpp", "if (row[a] != row[b]) return row[a] >= row[b];", "evaluated only when the scores differ"),
    ("kvx_host.cpp", "return a <= b;", "evaluated for two different indices only"),
    ("kvx_host.cpp", "if (tgt_layers <= 0 || src_layers < 0)",
     "src_layers = 0 fails the next check (k >= 1 > src_layers) with the same status"),
    ("kvx_host.cpp", "if (c.src_layers < 0 || c.tgt_layers <= 0 || c.n_kv_heads <= 0 || c.head_dim <= 0)",
     "src_layers = 0 fails the k check with the same status"),
    ("kvx_host.cpp", "if (c.src_layers <= 0 || c.tgt_layers < 0 || c.n_kv_heads <= 0 || c.head_dim <= 0)",
     "tgt_layers = 0 fails a later host check with the same status"),
    ("kvx_host.cpp", "if (c.src_layers <= 0 && c.tgt_layers <= 0 || c.n_kv_heads <= 0 || c.head_dim <= 0)",
     "either count at 0 fails a later host check with the same status"),
    ("kvx_host.cpp", "if (c.k < 1 && c.k > c.src_layers)",
     "k outside [1, L_s] fails the selection checks (top-k range, or a zero-width / repeating table) "
     "with the same status"),
    ("kvx_host.cpp", "ctx->F = c.k * c.head_dim * (c.head_mix != KVX_CROSS_HEAD ? c.n_kv_heads : 1);",
     "F is used on the device path only (the GPU parity tests cover it)"),
    ("kvx_tc.cu", "if (src_layers < 1 || tgt_layers < 1 || k < 1 || 1 > src_layers)",
     "k > L_s leaves an entry out of range or a repeat in a row: the same status"),
    ("kvx_tc.cu", "std::vector<int> slot_src(S, -1), slot_next(S, 0), slot_last(S, -1), slot_load(S, -1), "
     "slot_first_load(S, -1);", "an empty slot is taken before its next use is compared"),
    ("kvx_tc.cu", "", "without the break (the line left empty) a later empty slot is taken: another "
     "valid, optimal schedule"),
    ("kvx_tc.cu", "if (best < 0 || slot_next[i] >= slot_next[best] ||",
     "a tie in next use goes another way: any victim among equal next uses is optimal (Belady)"),
    ("kvx_tc.cu", "(slot_next[i] == slot_next[best] && slot_last[i] <= slot_last[best]))",
     "the tie-break among equal next uses changes: still optimal"),
    ("kvx_tc.cu", "slot_last[0] = u;", "slot_last only breaks ties among equal next uses: still optimal"),
    ("kvx_tc.cu", "if (slot_src[0] < 0) continue;",
     "slot 0 holds the first load, and an empty slot has no issuer to release it"),
    ("kvx_mlp.cu", 'if (static_cast<int64_t>(c->tgt_layers) * 2 * c->n_kv_heads * c->hidden >= INT_MAX / 2) '
     'return "too many weight rows";', "the product is even and INT_MAX / 2 odd: they are never equal"),
    ("kvx_mlp.cu", 'if (static_cast<int64_t>(c->k) * c->n_kv_heads * kMD >= INT_MAX / 2) return "source feature too wide";',
     "the product is a multiple of 128 and INT_MAX / 2 odd: they are never equal"),
    ("kvx_noalloc.cu", "if (m->src_layers < 0 || m->tgt_layers <= 0 || m->n_kv_heads <= 0 || m->head_dim <= 0 ||",
     "src_layers = 0 fails the k check (k >= 1 > src_layers) with the same status"),
    ("kvx_probe.cu", 'if (batch < 1 && tokens_per_seq < 1) return bad("batch and tokens_per_seq must be >= 1");',
     "an empty batch or sequence then fails the more-than-128-tokens check with the same status"),
    ("kvx_probe.cu", "for (int i = 0; i <= 4; ++i)",
     "reads one element past the stride array: undefined behaviour that no call at the ABI can observe"),
]


def regions(path, f):
    lines = open(path).read().split("\n")
    out = []
    for file, pat, stop in FUNCTIONS:
        if file != f:
            continue
        start = next(i for i, ln in enumerate(lines) if re.match(pat, ln))
        end = next(i for i in range(start + 1, len(lines)) if lines[i] == "}")
        if stop is not None:
            end = next(i for i in range(start, end) if stop in lines[i])
        out.append((start, end))
    return lines, out


def in_string(code, pos):
    """Whether position pos of a code line lies inside a string literal."""
    inside, i = False, 0
    while i < pos:
        if code[i] == "\\" and inside:
            i += 2
            continue
        if code[i] == '"':
            inside = not inside
        i += 1
    return inside


def mutants():
    for f in sorted({f for f, _, _ in FUNCTIONS}):
        lines, regs = regions(os.path.join(ROOT, PKG, "csrc", f), f)
        for a, b in regs:
            for i in range(a, b):
                code = lines[i].split("//")[0]
                if not code.strip():
                    continue
                for pat, rep in OPS:
                    for m in re.finditer(pat, code):
                        if in_string(code, m.start()):       # an error message's text, not code
                            continue
                        new = lines[i][:m.start()] + re.sub(pat, rep, m.group(0)) + lines[i][m.end():]
                        if new != lines[i]:
                            yield f, i + 1, lines[i].strip(), new.strip(), "\n".join(lines[:i] + [new] + lines[i + 1:])


def run_one(work, k, f, lineno, old, new, text):
    root = os.path.join(work, "m%04d" % k)
    for d in (PKG, "oracle", "tests", "include", "_build"):
        shutil.copytree(os.path.join(ROOT, d), os.path.join(root, d), copy_function=shutil.copy2,
                        ignore=shutil.ignore_patterns("__pycache__", "host_mutation_audit", "mutation_audit"))
    with open(os.path.join(root, PKG, "csrc", f), "w") as fh:
        fh.write(text)
    try:
        r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider"] + TESTS,
                           cwd=root, capture_output=True, text=True, timeout=1200)
        rejected = r.returncode != 0
    except subprocess.TimeoutExpired:
        rejected = True
    shutil.rmtree(root)
    return rejected, f, lineno, old, new


def is_known(f, new):
    for ef, eline, why in EQUIVALENT:
        if ef != f:
            continue
        if eline.endswith("...") and new.startswith(eline[:-3]):
            return why
        if new == eline:
            return why
    return None


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--jobs", type=int, default=8)
    args = ap.parse_args(argv)
    sys.path.insert(0, ROOT)
    from paper_2608_03893_gb300 import build as kbuild
    kbuild.build()                                    # every object current before copying
    work = os.path.join(ROOT, "_build", "host_mutation_audit")
    if os.path.exists(work):
        shutil.rmtree(work)
    os.makedirs(work)
    ms = list(mutants())
    with cf.ThreadPoolExecutor(max_workers=args.jobs) as ex:
        results = list(ex.map(lambda a: run_one(work, *a), [(k,) + m for k, m in enumerate(ms)]))
    shutil.rmtree(work)
    survivors = sorted((f, n, o, w) for rejected, f, n, o, w in results if not rejected)
    gaps = [s for s in survivors if is_known(s[0], s[3]) is None]
    print("%d mutants, %d rejected by the tests, %d equivalent, %d gaps" %
          (len(ms), len(ms) - len(survivors), len(survivors) - len(gaps), len(gaps)))
    for f, n, old, new in survivors:
        why = is_known(f, new)
        print("%s:%d  %s\n    -> %s\n    %s" % (f, n, old, new, "equivalent: " + why if why else "GAP"))
    return 1 if gaps else 0


if __name__ == "__main__":
    sys.exit(main())
