"""Pins for oracle.mapper (CPU only).

The paper prints no worked example of a mapping, so the mapping is pinned by:
* brute force: scalar Python loops over one output element at a time that write the
  RoPE as the complex product of Su et al. (an independent formulation of Sec. 3.3),
  for per-head and cross-head features, both pair layouts and both rounding models;
* closed forms: k = 1, W = I, b = 0 and equal thetas returns the source cache; with
  different thetas each pair turns by t (omega_t - omega_s); W = 0 gives
  K = R_t(t) b and V = b (the bias sits inside the re-rotated bracket of Sec. 3.3);
* invariants: linearity in W and b, per-head equals cross-head with W zero outside
  head h's rows, permuting the selection together with W's row blocks, and
  per-token independence (mapping a subset of tokens equals slicing the full map).
"""
import cmath
import math

import numpy as np
import pytest

from oracle import bf16, mapper, rope


def _problem(seed, Ls=3, Lt=4, H=2, N=6, d=8, k=2, head_mix="per_head", theta_s=1e4,
             theta_t=1e4):
    rng = np.random.default_rng(seed)
    src_k = rng.standard_normal((Ls, H, N, d))
    src_v = rng.standard_normal((Ls, H, N, d))
    pos = rng.integers(0, 5000, size=N)
    sel = np.sort(np.stack([rng.choice(Ls, size=k, replace=False) for _ in range(Lt)]), axis=1)
    F = k * d if head_mix == "per_head" else k * H * d
    W = rng.standard_normal((Lt, 2, H, F, d)) / math.sqrt(F)
    b = rng.standard_normal((Lt, 2, H, d)) * 0.1
    return dict(src_k=src_k, src_v=src_v, positions=pos, sel=sel, W=W, b=b,
                theta_s=theta_s, theta_t=theta_t)


def _pair_index(d, style):
    if style == "half":
        return [(i, i + d // 2) for i in range(d // 2)]
    return [(2 * i, 2 * i + 1) for i in range(d // 2)]


def _rot_scalar(vec, t, theta, sign, style):
    d = len(vec)
    out = list(vec)
    for i, (a, b) in enumerate(_pair_index(d, style)):
        z = complex(vec[a], vec[b]) * cmath.exp(1j * sign * t * theta ** (-2.0 * i / d))
        out[a], out[b] = z.real, z.imag
    return out


def _brute_element(P, l, kv, h, n, c, style, head_mix, mode):
    """One output element by scalar loops."""
    d = P["src_k"].shape[-1]
    H = P["src_k"].shape[1]
    t = int(P["positions"][n])
    feats = []
    for s in P["sel"][l]:
        heads = [h] if head_mix == "per_head" else list(range(H))
        for hh in heads:
            row = list(P["src_k"][s, hh, n] if kv == 0 else P["src_v"][s, hh, n])
            if kv == 0:
                row = _rot_scalar(row, t, P["theta_s"], -1, style)
                if mode == "bf16fwd":
                    row = [float(bf16.round_to_bf16_value(np.array([x]))[0]) for x in row]
            feats.extend(row)
    W = P["W"][l, kv, h]
    y = [sum(feats[f] * W[f, cc] for f in range(len(feats))) + P["b"][l, kv, h, cc]
         for cc in range(d)]
    if kv == 0:
        y = _rot_scalar(y, t, P["theta_t"], +1, style)
    return y[c]


@pytest.mark.parametrize("style", ["half", "interleaved"])
@pytest.mark.parametrize("head_mix", ["per_head", "cross_head"])
@pytest.mark.parametrize("mode", ["exact", "bf16fwd"])
def test_brute_force_elements(style, head_mix, mode):
    P = _problem(31, head_mix=head_mix, theta_s=1e4, theta_t=5e5)
    ok, ov = mapper.map_tokens(**P, mode=mode, style=style, head_mix=head_mix)
    rng = np.random.default_rng(32)
    Lt, H, N, d = ok.shape
    for _ in range(40):
        l, kv, h, n, c = (int(rng.integers(0, m)) for m in (Lt, 2, H, N, d))
        ref = _brute_element(P, l, kv, h, n, c, style, head_mix, mode)
        got = (ok if kv == 0 else ov)[l, h, n, c]
        assert abs(got - ref) < 1e-12 * max(1.0, abs(ref))


def test_identity_map_returns_source():
    P = _problem(33, k=1)
    d = P["src_k"].shape[-1]
    P["W"][:] = np.eye(d)
    P["b"][:] = 0.0
    P["sel"] = np.array([[0], [2], [1], [2]])
    ok, ov = mapper.map_tokens(**P)
    for l, s in enumerate(P["sel"][:, 0]):
        assert np.max(np.abs(ok[l] - P["src_k"][s])) < 1e-13
        assert np.array_equal(ov[l], P["src_v"][s])


def test_identity_map_different_thetas_closed_form():
    P = _problem(34, k=1, theta_s=1e4, theta_t=1e6)
    H, N, d = P["src_k"].shape[1:]
    P["W"][:] = np.eye(d)
    P["b"][:] = 0.0
    ok, _ = mapper.map_tokens(**P)
    i = np.arange(d // 2)
    dw = 1e6 ** (-2.0 * i / d) - 1e4 ** (-2.0 * i / d)
    for l, s in enumerate(P["sel"][:, 0]):
        x = P["src_k"][s]
        z = (x[..., : d // 2] + 1j * x[..., d // 2:]) * np.exp(1j * P["positions"][None, :, None] * dw)
        assert np.max(np.abs(ok[l] - np.concatenate([z.real, z.imag], -1))) < 1e-12


def test_zero_weights_give_rotated_bias():
    P = _problem(35)
    P["W"][:] = 0.0
    ok, ov = mapper.map_tokens(**P)
    d = ok.shape[-1]
    t = P["positions"]
    for l in range(ok.shape[0]):
        for h in range(ok.shape[1]):
            bk = P["b"][l, 0, h]
            for n in range(ok.shape[2]):
                expect = _rot_scalar(list(bk), int(t[n]), P["theta_t"], +1, "half")
                assert np.max(np.abs(ok[l, h, n] - expect)) < 1e-14
            assert np.array_equal(ov[l, h], np.broadcast_to(P["b"][l, 1, h], (ok.shape[2], d)))


def test_linearity_in_weights_and_bias():
    P1, P2 = _problem(36), _problem(37)
    P2.update(src_k=P1["src_k"], src_v=P1["src_v"], positions=P1["positions"], sel=P1["sel"])
    a, c = 0.37, -1.9
    P3 = dict(P1, W=a * P1["W"] + c * P2["W"], b=a * P1["b"] + c * P2["b"])
    k1, v1 = mapper.map_tokens(**P1)
    k2, v2 = mapper.map_tokens(**P2)
    k3, v3 = mapper.map_tokens(**P3)
    assert np.max(np.abs(k3 - (a * k1 + c * k2))) < 1e-12
    assert np.max(np.abs(v3 - (a * v1 + c * v2))) < 1e-12


def test_per_head_equals_cross_head_with_block_weights():
    P = _problem(38, head_mix="per_head")
    Lt, _, H, F, d = P["W"].shape
    k = F // d
    Wc = np.zeros((Lt, 2, H, k * H * d, d))
    for j in range(k):
        for h in range(H):
            Wc[:, :, h, (j * H + h) * d:(j * H + h + 1) * d] = P["W"][:, :, h, j * d:(j + 1) * d]
    kp, vp = mapper.map_tokens(**P, head_mix="per_head")
    kc, vc = mapper.map_tokens(**dict(P, W=Wc), head_mix="cross_head")
    assert np.max(np.abs(kp - kc)) < 1e-12 and np.max(np.abs(vp - vc)) < 1e-12


def test_selection_permutation_with_weight_blocks():
    P = _problem(39, k=3, Ls=4)
    d = P["src_k"].shape[-1]
    perm = [2, 0, 1]
    Wp = np.concatenate([P["W"][..., j * d:(j + 1) * d, :] for j in perm], axis=-2)
    k1, v1 = mapper.map_tokens(**P)
    k2, v2 = mapper.map_tokens(**dict(P, sel=P["sel"][:, perm], W=Wp))
    assert np.max(np.abs(k1 - k2)) < 1e-12 and np.max(np.abs(v1 - v2)) < 1e-12


def test_per_token_independence():
    P = _problem(40, N=9)
    k_all, v_all = mapper.map_tokens(**P)
    idx = np.array([7, 2, 5])
    Q = dict(P, src_k=P["src_k"][:, :, idx], src_v=P["src_v"][:, :, idx], positions=P["positions"][idx])
    k_sub, v_sub = mapper.map_tokens(**Q)
    assert np.array_equal(k_sub, k_all[:, :, idx]) and np.array_equal(v_sub, v_all[:, :, idx])


def test_bf16fwd_equals_exact_when_stripped_keys_are_bf16():
    # at position 0 the strip is the identity, so bf16 inputs stay bf16: both modes agree
    P = _problem(41)
    P["src_k"] = bf16.round_to_bf16_value(P["src_k"])
    P["positions"] = np.zeros_like(P["positions"])
    ke, ve = mapper.map_tokens(**P, mode="exact")
    kb, vb = mapper.map_tokens(**P, mode="bf16fwd")
    assert np.array_equal(ke, kb) and np.array_equal(ve, vb)


def test_bf16fwd_error_bounded_by_operand_rounding():
    P = _problem(42, N=20)
    ke, _ = mapper.map_tokens(**P, mode="exact")
    kb, _ = mapper.map_tokens(**P, mode="bf16fwd")
    # |dX| <= 2^-9 |X| per element; rotation is orthogonal: |dy| <= 2^-9 sum|X||W| per pair norm
    Xmax = np.max(np.abs(P["src_k"])) * math.sqrt(2)
    F = P["W"].shape[-2]
    bound = 2.0 ** -9 * Xmax * np.max(np.abs(P["W"])) * F * math.sqrt(2)
    diff = np.max(np.abs(ke - kb))
    assert 0 < diff < bound


def test_map_cache_layout_roundtrip():
    rng = np.random.default_rng(43)
    Ls, Lt, B, H, T, d, k = 3, 3, 2, 2, 5, 8, 2           # L_t, B, H, T all different
    B = 4
    src_k = rng.standard_normal((Ls, B, H, T, d))
    src_v = rng.standard_normal((Ls, B, H, T, d))
    pos = np.stack([np.arange(T) + 100 * bb for bb in range(B)])
    sel = np.array([[0, 2], [1, 2], [0, 1]])
    W = rng.standard_normal((Lt, 2, H, k * d, d))
    b = rng.standard_normal((Lt, 2, H, d))
    for kw in ({}, dict(mode="bf16fwd", style="interleaved"), dict(rope_numerics="hf")):
        ck, cv = mapper.map_cache(src_k, src_v, pos, sel, W, b, 1e4, 5e5, **kw)
        for bb in range(B):
            tk, tv = mapper.map_tokens(src_k[:, bb], src_v[:, bb], pos[bb], sel, W, b, 1e4, 5e5, **kw)
            assert np.array_equal(ck[:, bb], tk) and np.array_equal(cv[:, bb], tv)
    # and the thetas and the mode reach the map: other values give another cache
    ck2, _ = mapper.map_cache(src_k, src_v, pos, sel, W, b, 5e5, 1e4)
    ck3, _ = mapper.map_cache(src_k, src_v, pos, sel, W, b, 1e4, 5e5, mode="bf16fwd")
    assert not np.array_equal(ck, ck2) and not np.array_equal(ck, ck3)


def test_rounding_slack_is_zero_without_ambiguity_and_for_values():
    P = _problem(44, N=10)
    ok, ov, sk, sv = mapper.map_tokens(**P, mode="bf16fwd", rounding_slack=0.0)
    assert np.all(sk == 0) and np.all(sv == 0)
    ok2, ov2, sk2, sv2 = mapper.map_tokens(**P, mode="bf16fwd", rounding_slack=4e-6)
    assert np.array_equal(ok, ok2) and np.all(sv2 == 0)
    # the slack leaves the mapped cache itself unchanged, keys and values
    ok0, ov0 = mapper.map_tokens(**P, mode="bf16fwd")
    assert np.array_equal(ok0, ok2) and np.array_equal(ov0, ov2) and np.array_equal(ov0, ov)
    assert not np.array_equal(ok0, ov0)


def test_rounding_slack_covers_both_roundings_of_a_planted_midpoint():
    """Content keys sitting exactly on a bf16 midpoint are rotated into the cache; the
    oracle's f64 strip lands within 1e-15 of the midpoint and may round either way.
    Both choices, evaluated directly, must lie within out +- slack."""
    rng = np.random.default_rng(45)
    Ls, Lt, H, N, d, k = 3, 2, 2, 3, 8, 2
    # |content| in [0.5, 2]: a stored pair's fp32-strip uncertainty (4e-6 of |a| + |b|)
    # stays far below half a bf16 step of either element, so the planted midpoints are
    # the only ambiguous roundings
    content = bf16.round_to_bf16_value(rng.choice([-1.0, 1.0], size=(Ls, H, N, d)) *
                                       rng.uniform(0.5, 2.0, size=(Ls, H, N, d)))
    # midpoints only in head 1: of source layer 0 (channel 1) and source layer 1 (channel 6)
    content[0, 1, :, 1] = 1.0 + 2.0 ** -8          # ties between 1 and 1 + 2^-7
    content[1, 1, :, 6] = -(3.0 + 2.0 ** -7)        # ties between -3 and -(3 + 2^-6)
    pos = np.array([0, 77, 30001])
    stored = np.stack([rope.rotate(content[s], pos[None, :], 1e4) for s in range(Ls)])
    sel = np.array([[0, 2], [1, 2]])               # each target layer meets one planted layer
    W = rng.standard_normal((Lt, 2, H, k * d, d)) / 4
    b = rng.standard_normal((Lt, 2, H, d)) * 0.1
    src_v = rng.standard_normal((Ls, H, N, d))
    out_k, out_v, slack_k, slack_v = mapper.map_tokens(stored, src_v, pos, sel, W, b, 1e4, 1e4,
                                                       mode="bf16fwd", rounding_slack=4e-6)
    for down in (True, False):
        X = content.copy()
        X[0, 1, :, 1] = 1.0 if down else 1.0 + 2.0 ** -7
        X[1, 1, :, 6] = -3.0 if down else -(3.0 + 2.0 ** -6)
        for l in range(Lt):
            for h in range(H):
                Xl = np.concatenate([X[s, h] for s in sel[l]], axis=-1)
                y = rope.rotate(Xl @ W[l, 0, h] + b[l, 0, h], pos, 1e4)
                assert np.all(np.abs(y - out_k[l, h]) <= slack_k[l, h] + 1e-12)
    assert np.all(slack_k[:, 1] > 0)     # every output of head 1 meets a planted pair
    assert np.all(slack_k[:, 0] == 0) and np.all(slack_v == 0)
    # the slack is the worst case of the other rounding: |W| rows of the ambiguous feature
    # (feature 1 of block 0 in layer 0, feature 6 of block 0 in layer 1), its bf16 step
    # (2^-7 and 2^-6), summed over the output's RoPE pair after the rotation
    for l, f, step in ((0, 1, 2.0 ** -7), (1, 6, 2.0 ** -6)):
        per_c = step * np.abs(W[l, 0, 1, f])                  # [d]
        want = np.concatenate([per_c[:4] + per_c[4:]] * 2)
        assert np.allclose(slack_k[l, 1], np.broadcast_to(want, (N, d)), rtol=1e-12, atol=0)
    # cross-head features with W zero outside head h's rows give the same map and slack
    Wx = np.zeros((Lt, 2, H, k * H * d, d))
    for l in range(Lt):
        for h in range(H):
            for j in range(k):
                Wx[l, :, h, (j * H + h) * d:(j * H + h + 1) * d] = W[l, :, h, j * d:(j + 1) * d]
    xk, xv, xsk, xsv = mapper.map_tokens(stored, src_v, pos, sel, Wx, b, 1e4, 1e4, mode="bf16fwd",
                                         rounding_slack=4e-6, head_mix="cross_head")
    assert np.allclose(xk, out_k, rtol=0, atol=1e-12) and np.allclose(xv, out_v, rtol=0, atol=1e-12)
    assert np.allclose(xsk, slack_k, rtol=1e-12, atol=0) and np.all(xsv == 0)


def test_slack_helpers_hand_values():
    x = np.array([1.0, -2.0, 3.0, -4.0])
    # half-split pairs (0, 2), (1, 3); interleaved pairs (0, 1), (2, 3)
    assert mapper._pair_magnitude(x, "half").tolist() == [4.0, 6.0, 4.0, 6.0]
    assert mapper._pair_magnitude(x, "interleaved").tolist() == [3.0, 3.0, 7.0, 7.0]
    assert mapper._pair_magnitude(-x, "half").tolist() == [4.0, 6.0, 4.0, 6.0]
    assert mapper._pair_magnitude(-x, "interleaved").tolist() == [3.0, 3.0, 7.0, 7.0]
    assert mapper._pair_sum(x, "half").tolist() == [4.0, -6.0, 4.0, -6.0]
    assert mapper._pair_sum(x, "interleaved").tolist() == [-1.0, -1.0, -1.0, -1.0]


def test_unknown_mode_is_rejected():
    with pytest.raises(ValueError):
        mapper.map_tokens(**_problem(48), mode="fp8")


@pytest.mark.parametrize("style", ["half", "interleaved"])
def test_hf_numerics_identity_map_returns_the_source_keys(style):
    """k = 1, W = I, b = 0, equal thetas with the Hugging Face rounding: the strip and
    the re-rotation cancel up to the bf16 roundings of the two rotations (each product,
    sum and cos / sin rounded once: well under 2^-5 of the pair magnitude), on caches
    whose L, H, N and d all differ."""
    rng = np.random.default_rng(47)
    Ls, H, N, d = 2, 3, 7, 16
    src_k = bf16.round_to_bf16_value(rng.standard_normal((Ls, H, N, d)))
    src_v = bf16.round_to_bf16_value(rng.standard_normal((Ls, H, N, d)))
    pos = np.array([1, 5, 77, 300, 4000, 30001, 65535])
    sel = np.array([[1], [0]])
    W = np.broadcast_to(np.eye(d), (2, 2, H, d, d)).copy()
    for mode in ("exact", "bf16fwd"):
        ok, ov = mapper.map_tokens(src_k, src_v, pos, sel, W, None, 5e5, 5e5, mode=mode, style=style,
                                   rope_numerics="hf")
        for l, s in ((0, 1), (1, 0)):
            mag = mapper._pair_magnitude(src_k[s], style)
            assert np.all(np.abs(ok[l] - src_k[s]) <= 2.0 ** -5 * mag + 1e-30)
            assert np.array_equal(ov[l], src_v[s])
        # the HF rounding is visible: not the exact-numerics result
        ek, _ = mapper.map_tokens(src_k, src_v, pos, sel, W, None, 5e5, 5e5, mode=mode, style=style)
        assert not np.array_equal(ok, ek)
