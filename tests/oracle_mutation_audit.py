"""Mutation audit of the oracle's pins (CPU; run by hand, not collected by pytest).

Each mutant changes one operator on one code line of ``oracle/*.py`` (a sign, an index,
an axis, a comparison, a constant, cos for sin, a reduction, an argument such as theta_s
for theta_t, a rounding point such as float32 for float64) in a private copy of the
package, and runs the oracle pin tests against it.  A mutant the pins do not reject is a
"survivor".  Survivors listed in EQUIVALENT compute the same result on every input the
oracle accepts, for the reason given; any other survivor is a gap in the pins and makes
the audit exit with status 1.

    python tests/oracle_mutation_audit.py [--jobs 6]

Copies go under ``_build/mutation_audit/`` (git-ignored) and are removed afterwards.
"""
import argparse
import concurrent.futures as cf
import os
import re
import shutil
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PIN_TESTS = ["tests/test_oracle_rope.py", "tests/test_oracle_mapper.py", "tests/test_oracle_fit.py",
             "tests/test_oracle_mlp.py"]

OPS = [
    (r" \+ ", " - "), (r" - ", " + "), (r"\bcos\b", "sin"), (r"\bsin\b", "cos"),
    (r"axis=0", "axis=1"), (r"axis=1", "axis=0"), (r"\.T\b", ""), (r" < ", " <= "), (r" > ", " >= "),
    (r" <= ", " < "), (r" >= ", " > "), (r"\[0\]", "[1]"), (r"\[1\]", "[0]"), (r"\b0\.5\b", "0.25"),
    (r"\b2\.0\b", "1.0"), (r"\b1\.0\b", "2.0"), (r"-1\b", "1"), (r"\b2 \* ", ""), (r" \* 2\b", ""),
    (r"\bmin\(", "max("), (r"\bmax\(", "min("), (r"\bh\b", "0"), (r"\bl\b", "0"), (r"\bj\b", "0"),
    (r"np\.sum\(", "np.mean("), (r"np\.mean\(", "np.sum("), (r"\+= ", "= "), (r"\bTrue\b", "False"),
    (r"// 2\b", "// 4"), (r"- 1\b", ""), (r"\+ 1\b", ""),
    (r"\btheta_s\b", "theta_t"), (r"\btheta_t\b", "theta_s"), (r"np\.abs\(", "("), (r"0::2", "1::2"),
    (r"1::2", "0::2"), (r"-2\.0", "2.0"), (r"\.mean\(", ".sum("), (r"\.sum\(", ".mean("),
    (r"\bnp\.rint\(", "np.floor("), (r"\bsqrt\(", "abs("), (r"\blower=True\b", "lower=False"),
    (r"\bstyle=style\b", "style=\"half\""), (r"\bbf16_cache=True\b", "bf16_cache=False"),
    (r"\bmode\b", "\"exact\""), (r"\[::-1\]", ""), (r"\bx_mean\b", "0.0"), (r"\by_mean\b", "0.0"),
    (r"\blam\b", "lam2"), (r"\bnp\.float32\b", "np.float64"),
    (r"axis=-1", "axis=0"), (r"\[None, :\]", "[:, None]"), (r"\[:, None\]", "[None, :]"),
    (r"\brange\((\w+)\)", "range(1)"), (r"\*\* 2\b", "** 1"), (r": d // 2\]", "d // 2:]"),
    (r"\bd // 2:\]", ": d // 2]"),
]

# (file, mutated line after the change, why it computes the same result)
EQUIVALENT = [
    ("bf16.py", "small = e - 1 <= _MIN_NORMAL_EXP",
     "at e - 1 = -126 both quanta are 2^-133 (e - 8 = -133), so the boundary value rounds alike"),
    ("mapper.py", "X = np.concatenate(parts, axis=1)", "parts are 2-D [N][d]: axis 1 is the last axis"),
    ("mapper.py", "A = np.concatenate([amb[s, h] for s in sel[l]], axis=1)", "2-D parts: axis 1 is the last"),
    ("mapper.py", "A = np.concatenate([amb[s, hh] for s in sel[l] for hh in range(H)], axis=1)",
     "2-D parts: axis 1 is the last"),
    ("mapper.py", "Lt = res[1].shape[0]", "keys and values have the same L_t"),
    ("mlp.py", "parts.append(np.concatenate(list(x), axis=1))      # [N][H d], head-minor",
     "each head's slice is 2-D [N][d]: axis 1 is the last"),
    ("mlp.py", "return np.concatenate(parts, axis=1)", "2-D parts: axis 1 is the last"),
    ("ridge.py", "Yc = Y + y_mean",
     "W only sees Xc^T Yc and Xc^T 1 = 0 (X is centred), so the sign of the Y mean drops out; b uses y_mean itself"),
    ("ridge.py", "Yc = Y - 0.0", "as above: Xc^T Y = Xc^T Yc for a centred Xc"),
    ("rope.py", "ang = (p32[..., None] * w32).astype(np.float64).astype(np.float64)   # fp32 multiply, rounded",
     "p32 and w32 are float32 arrays, so numpy's product is already the binary32 product"),
    ("mapper.py", 'raise ValueError("exact")', "only the error message's text changes"),
    ("ridge.py", "factor = scipy.linalg.cho_factor(A, lower=False)",
     "cho_solve follows the factor's own lower / upper flag"),
    ("rope.py", "out = np.where(lam <= P / s.high_freq_factor, omega, blend)",
     "the Llama-3 blend equals omega at that band edge (continuity, pinned)"),
    ("rope.py", "return np.where(lam >= P / s.low_freq_factor, omega / s.factor, out)",
     "the Llama-3 blend equals omega / factor at that band edge (continuity, pinned)"),
]


def code_lines(text):
    """Indices of lines that are code (not docstring, comment or blank)."""
    out, in_doc = [], False
    for i, ln in enumerate(text.split("\n")):
        st = ln.strip()
        q = st.count('"""')
        if in_doc:
            if q % 2 == 1:
                in_doc = False
            continue
        if st.startswith('"""'):
            if q == 1:
                in_doc = True
            continue
        if st and not st.startswith("#"):
            out.append(i)
    return out


def mutants():
    src = os.path.join(ROOT, "oracle")
    for f in sorted(os.listdir(src)):
        if not f.endswith(".py") or f == "__init__.py":
            continue
        lines = open(os.path.join(src, f)).read().split("\n")
        for i in code_lines("\n".join(lines)):
            code = lines[i].split("#")[0]
            for pat, rep in OPS:
                for m in re.finditer(pat, code):
                    new = lines[i][:m.start()] + re.sub(pat, rep, m.group(0)) + lines[i][m.end():]
                    if new != lines[i]:
                        yield f, i + 1, lines[i].strip(), new.strip(), "\n".join(lines[:i] + [new] + lines[i + 1:])


def run_one(work, k, f, lineno, old, new, text):
    root = os.path.join(work, "m%04d" % k)
    shutil.copytree(os.path.join(ROOT, "oracle"), os.path.join(root, "oracle"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    shutil.copytree(os.path.join(ROOT, "tests"), os.path.join(root, "tests"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    os.symlink(os.path.join(ROOT, "paper_2608_03893_gb300"), os.path.join(root, "paper_2608_03893_gb300"))
    with open(os.path.join(root, "oracle", f), "w") as fh:
        fh.write(text)
    try:
        r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider"] + PIN_TESTS,
                           cwd=root, capture_output=True, text=True, timeout=300)
        rejected = r.returncode != 0
    except subprocess.TimeoutExpired:
        rejected = True
    shutil.rmtree(root)
    return rejected, f, lineno, old, new


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--jobs", type=int, default=6)
    args = ap.parse_args(argv)
    work = os.path.join(ROOT, "_build", "mutation_audit")
    if os.path.exists(work):
        shutil.rmtree(work)
    os.makedirs(work)
    ms = list(mutants())
    with cf.ThreadPoolExecutor(max_workers=args.jobs) as ex:
        results = list(ex.map(lambda a: run_one(work, *a), [(k,) + m for k, m in enumerate(ms)]))
    shutil.rmtree(work)
    survivors = sorted((f, n, o, w) for rejected, f, n, o, w in results if not rejected)
    known = {(f, new): why for f, new, why in EQUIVALENT}
    gaps = [s for s in survivors if (s[0], s[3]) not in known]
    print("%d mutants, %d rejected by the pins, %d equivalent, %d gaps" %
          (len(ms), len(ms) - len(survivors), len(survivors) - len(gaps), len(gaps)))
    for f, n, old, new in survivors:
        tag = "equivalent: " + known[(f, new)] if (f, new) in known else "GAP"
        print("%s:%d  %s\n    -> %s\n    %s" % (f, n, old, new, tag))
    return 1 if gaps else 0


if __name__ == "__main__":
    sys.exit(main())
