"""Host side of __graft_entry__.smoke() (no GPU): the error report it prints."""
import numpy as np

import __graft_entry__ as entry
from oracle import bf16 as obf16
from oracle import mapper as omap
from oracle import selection as osel
from paper_2608_03893_gb300 import synthetic as syn


def test_error_report_on_planted_errors():
    rng = np.random.default_rng(0)
    rk = rng.standard_normal((3, 1, 2, 4, 8))
    rv = rng.standard_normal((3, 1, 2, 4, 8))
    rms = np.sqrt(np.mean(np.concatenate([rk.ravel(), rv.ravel()]) ** 2))
    gk, gv = rk.copy(), rv.copy()
    gv[2, 0, 1, 3, 5] += 0.25                      # one error, in V of target layer 2
    rep = entry.error_report(gk, gv, rk, rv, rk, rv)
    assert abs(rep["bf16fwd"] - 0.25 / rms) < 1e-12 and rep["exact"] == rep["bf16fwd"]
    assert rep["worst_slice_at"] == (2, "V")
    assert abs(rep["worst_slice"] - 0.25 / np.sqrt(np.mean(rv[2] ** 2))) < 1e-12
    # the exact-mode reference enters only the "exact" figure
    ek = rk + 0.5
    rep = entry.error_report(gk, gv, rk, rv, ek, rv)
    assert abs(rep["exact"] - 0.5 / rms) < 1e-12 and abs(rep["bf16fwd"] - 0.25 / rms) < 1e-12


def test_error_report_at_the_smoke_shape():
    # the oracle calls smoke() makes, with a device output that is the bf16-forward
    # result rounded once to bf16 (what a correct kernel produces up to the slack)
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=6, Lt=5, H=2, B=2, T=200, k=3)
    W, b = syn.weights(w)
    sel = osel.select_topk(syn.selection_scores(w), w.k)

    def f64(t):
        return obf16.decode(t.contiguous().view(__import__("torch").int16).numpy().view(np.uint16))

    sk, sv = syn.source_cache(w, 0), syn.source_cache(w, 1)
    rk, rv, ak, av = omap.map_cache(f64(sk), f64(sv), syn.positions(w), sel, f64(W), f64(b),
                                    w.theta_s, w.theta_t, mode="bf16fwd", rounding_slack=4e-6)
    ek, ev = omap.map_cache(f64(sk), f64(sv), syn.positions(w), sel, f64(W), f64(b),
                            w.theta_s, w.theta_t, mode="exact")
    gk, gv = obf16.round_to_bf16_value(rk), obf16.round_to_bf16_value(rv)
    rep = entry.error_report(gk, gv, rk, rv, ek, ev)
    rms = np.sqrt(np.mean(np.concatenate([rk.ravel(), rv.ravel()]) ** 2))
    peak = max(np.max(np.abs(rk)), np.max(np.abs(rv))) / rms
    assert 0 < rep["bf16fwd"] <= 2.0 ** -8 * peak           # one bf16 rounding of the output
    # values are exact bf16 in both modes; keys differ by the rounding of the stripped
    # operand, of the order of 2^-8 of the output RMS
    assert rep["bf16fwd"] <= rep["exact"] < 0.05
    assert rep["worst_slice_at"][0] in range(w.Lt) and rep["worst_slice_at"][1] in ("K", "V")
