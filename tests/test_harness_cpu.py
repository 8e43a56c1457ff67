"""The comparison the GPU parity tests use (tests/harness.py), checked on CPU arrays:
the stated tolerances, the rounding slack for bf16 only, NaN as a failure, and the rows
the full-size tests sample."""
import numpy as np

import harness as H
from paper_2608_03893_gb300 import synthetic as syn


def test_tolerance_constants_are_the_stated_ones():
    assert H.F32_ABS_RMS == 1e-4 and H.BF16_REL == 2.0 ** -7 and H.BF16_ABS_RMS == 1e-3
    assert H.STRIP_DELTA == 4e-6


def _ref():
    rng = np.random.default_rng(3)
    return [rng.standard_normal((2, 3, 5, 8)), rng.standard_normal((2, 3, 5, 8))]


def test_bf16_bound_from_both_sides():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4")
    ref = _ref()
    r = np.concatenate([x.ravel() for x in ref])
    rms = np.sqrt(np.mean(r * r))
    i = int(np.argmax(np.abs(ref[1])))                # one element of V
    bound = 2.0 ** -7 * abs(ref[1].flat[i]) + 1e-3 * rms
    for scale, ok in ((0.999, True), (1.001, False)):
        got = [x.copy() for x in ref]
        got[1].flat[i] += scale * bound
        res = H.check(w, got, ref)
        assert res[0] is ok and res[3] == (0 if ok else 1), scale
        assert abs(res[1] - scale) < 1e-9 and abs(res[2] - rms) < 1e-12
    # the slack widens exactly that element's bound, and only on bf16 workloads
    got = [x.copy() for x in ref]
    got[1].flat[i] += 1.5 * bound
    slack = [np.zeros_like(x) for x in ref]
    slack[1].flat[i] = 0.5 * bound
    assert H.check(w, got, ref, slack)[0] is False
    slack[1].flat[i] = 0.51 * bound
    assert H.check(w, got, ref, slack)[0] is True
    # a NaN fails
    got = [x.copy() for x in ref]
    got[0].flat[3] = np.nan
    res = H.check(w, got, ref)
    assert res[0] is False and res[3] == 1 and res[1] == float("inf")


def test_f32_bound_from_both_sides():
    w = syn.workload("tiny_fp32")
    ref = _ref()
    r = np.concatenate([x.ravel() for x in ref])
    rms = np.sqrt(np.mean(r * r))
    for scale, ok in ((0.999, True), (1.001, False)):
        got = [x.copy() for x in ref]
        got[0].flat[7] -= scale * 1e-4 * rms        # no relative term for fp32
        assert H.check(w, got, ref)[0] is ok, scale
    got = [x.copy() for x in ref]
    got[0].flat[7] -= 2e-4 * rms
    big = [np.full_like(x, 1.0) for x in ref]         # the slack is not used for fp32
    assert H.check(w, got, ref, big)[0] is False


def test_sampled_rows_cover_the_tile_borders_and_the_tail():
    w = syn.workload("qwen3_14b_32b_t32768_k4")
    rows = H.sample_rows(w, 40, seed=2)
    want = {(0, 0), (0, 1), (0, 127), (0, 128), (w.B - 1, w.T - 1), (w.B - 1, w.T - 2),
            (w.B - 1, (w.T - 1) // 128 * 128)}
    got = {tuple(r) for r in rows.tolist()}
    assert want <= got and len(got) >= 40 and len(got) == len(rows)
    assert rows[:, 0].min() >= 0 and rows[:, 0].max() < w.B and rows[:, 1].min() >= 0 and rows[:, 1].max() < w.T
    # a short sequence (fewer than 129 tokens) keeps only rows inside it
    rows = H.sample_rows(w, 5, turn_T=100)
    assert rows[:, 1].max() < 100 and (0, 127) not in {tuple(r) for r in rows.tolist()}
    # exactly one tile: nothing at t = 128; one token past a tile: that token's row is in
    rows = H.sample_rows(w, 5, turn_T=128)
    assert rows[:, 1].max() == 127
    rows = H.sample_rows(w, 5, turn_T=129)
    assert (w.B - 1, 128) in {tuple(r) for r in rows.tolist()}


def test_oracle_rows_are_the_rows_of_the_full_oracle():
    """The full-size parity tests compare sampled rows against oracle_rows; those must be
    exactly the corresponding rows of the full oracle map (both layouts, both modes, a
    Llama-3-scaled workload), addressed by (batch, token)."""
    from oracle import selection as osel
    cases = [syn.workload("tiny_fp32", B=3, T=40),
             syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=5, Lt=3, H=2, B=2, T=37, k=2, theta_t=5e5),
             syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=4, Lt=2, H=2, B=2, T=20, k=2, rope_style="interleaved"),
             syn.workload("llama31_8b_70b_b4x8192_k3", Ls=4, Lt=3, H=2, B=2, T=24, k=2,
                          rope_scaling=(8.0, 1.0, 4.0, 8192.0))]
    for w in cases:
        W, b = syn.weights(w)
        sel = osel.select_topk(syn.selection_scores(w), w.k)
        pos = syn.positions(w) * 1000 + 7                  # positions far from the token index
        rk, rv, ak, av = H.oracle_full(w, syn.source_cache(w, 0), syn.source_cache(w, 1), pos, sel, W, b)
        rows = np.array([[0, 0], [w.B - 1, w.T - 1], [1, 3], [0, w.T // 2]])
        ok, ov, sk, sv = H.oracle_rows(w, rows, pos, sel, W, b)
        for n, (bb, t) in enumerate(rows):
            assert np.array_equal(ok[:, :, n], rk[:, bb, :, t]) and np.array_equal(ov[:, :, n], rv[:, bb, :, t])
            assert np.array_equal(sk[:, :, n], ak[:, bb, :, t]) and np.array_equal(sv[:, :, n], av[:, bb, :, t])
        assert np.array_equal(H.to_f64(W), W.double().numpy())


def test_rope_theta_sides():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", theta_s=1e4, theta_t=5e5)
    assert (H.rope_theta(w, 0), H.rope_theta(w, 1)) == (1e4, 5e5)
    w = syn.workload("llama31_8b_70b_b4x8192_k3", theta_s=1e4, theta_t=5e5, rope_scaling=(8.0, 1.0, 4.0, 8192.0))
    s0, s1 = H.rope_theta(w, 0), H.rope_theta(w, 1)
    assert (s0.theta, s1.theta) == (1e4, 5e5)
    assert tuple(s0.scaling) == tuple(s1.scaling) == (8.0, 1.0, 4.0, 8192.0)
