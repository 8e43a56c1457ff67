"""Pins for oracle.rope and oracle.bf16 (CPU only).

RoPE is pinned against the complex-number definition of Su et al. (Sec. 3.3 cites it:
pair i is multiplied by exp(i t omega_i)), against a textbook 2x2 rotation matrix,
and by the group identities R(-t) R(t) = I, R(a) R(b) = R(a + b), R(0) = I and
orthogonality (pair norms preserved).  bf16 rounding is pinned against hand-worked
bit patterns and against torch's binary32 -> bfloat16 conversion.
"""
import math

import numpy as np
import pytest
import torch

from oracle import bf16, rope


def _rng(seed=0):
    return np.random.default_rng(seed)


@pytest.mark.parametrize("style", ["half", "interleaved"])
def test_inverse_is_identity(style):
    x = _rng(1).standard_normal((3, 5, 64))
    pos = _rng(2).integers(0, 40000, size=(3, 5))
    y = rope.rotate(rope.rotate(x, pos, 1e6, style=style), pos, 1e6, inverse=True, style=style)
    assert np.max(np.abs(y - x)) < 1e-12


@pytest.mark.parametrize("style", ["half", "interleaved"])
def test_pair_norms_preserved(style):
    d = 32
    x = _rng(3).standard_normal((7, d))
    pos = np.arange(7) * 4099
    y = rope.rotate(x, pos, 5e5, style=style)
    if style == "half":
        nx = x[:, : d // 2] ** 2 + x[:, d // 2:] ** 2
        ny = y[:, : d // 2] ** 2 + y[:, d // 2:] ** 2
    else:
        nx = x[:, 0::2] ** 2 + x[:, 1::2] ** 2
        ny = y[:, 0::2] ** 2 + y[:, 1::2] ** 2
    assert np.allclose(nx, ny, rtol=1e-13, atol=1e-13)


def test_position_zero_is_exact_identity():
    x = _rng(4).standard_normal((4, 128))
    y = rope.rotate(x, np.zeros(4, dtype=np.int64), 1e6)
    assert np.array_equal(x, y)
    y = rope.rotate(x, np.zeros(4, dtype=np.int64), 1e6, inverse=True)
    assert np.array_equal(x, y)


def test_angle_additivity():
    x = _rng(5).standard_normal((6, 64))
    a = np.array([0, 1, 17, 255, 1000, 32767])
    b = np.array([3, 0, 9, 1, 31000, 1])
    y1 = rope.rotate(rope.rotate(x, a, 1e4), b, 1e4)
    y2 = rope.rotate(x, a + b, 1e4)
    assert np.max(np.abs(y1 - y2)) < 1e-10


def test_complex_multiplication_definition():
    """Pair i of the half-split layout is (x[i] + 1j x[i+d/2]) * exp(1j t theta^(-2i/d))."""
    d, theta = 16, 10000.0
    x = _rng(6).standard_normal((9, d))
    pos = np.array([0, 1, 2, 5, 77, 1023, 4096, 20000, 32767])
    z = x[:, : d // 2] + 1j * x[:, d // 2:]
    w = np.array([[theta ** (-2.0 * i / d) for i in range(d // 2)]])
    zr = z * np.exp(1j * pos[:, None] * w)
    expect = np.concatenate([zr.real, zr.imag], axis=1)
    got = rope.rotate(x, pos, theta)
    assert np.max(np.abs(got - expect)) < 1e-12
    # the inverse multiplies by the conjugate
    zi = z * np.exp(-1j * pos[:, None] * w)
    got_i = rope.rotate(x, pos, theta, inverse=True)
    assert np.max(np.abs(got_i - np.concatenate([zi.real, zi.imag], axis=1))) < 1e-12


def test_first_pair_rotates_by_position_radians():
    """omega_0 = 1, so pair 0 rotates by exactly t radians: a textbook 2x2 rotation."""
    for t in [1, 3, 100, 32767]:
        a, b = 0.3, -1.7
        x = np.zeros((1, 8))
        x[0, 0], x[0, 4] = a, b
        y = rope.rotate(x, np.array([t]), 1e6)
        rot = np.array([[math.cos(t), -math.sin(t)], [math.sin(t), math.cos(t)]])
        ea, eb = rot @ np.array([a, b])
        assert abs(y[0, 0] - ea) < 1e-14 and abs(y[0, 4] - eb) < 1e-14


def test_half_and_interleaved_agree_under_permutation():
    d = 64
    x = _rng(7).standard_normal((5, d))
    pos = np.array([0, 3, 999, 12345, 32000])
    perm = np.empty(d, dtype=np.int64)  # interleaved index 2i <- half i, 2i+1 <- half i+d/2
    perm[0::2] = np.arange(d // 2)
    perm[1::2] = np.arange(d // 2) + d // 2
    yh = rope.rotate(x, pos, 1e6, style="half")
    yi = rope.rotate(x[:, perm], pos, 1e6, style="interleaved")
    assert np.max(np.abs(yh[:, perm] - yi)) < 1e-14


def test_inverse_frequencies():
    w = rope.inv_freq(1e6, 128)
    assert w[0] == 1.0
    assert abs(w[32] - 1e6 ** -0.5) < 1e-18
    assert abs(w[63] / w[62] - 1e6 ** (-2.0 / 128)) < 1e-14


# ---------------------------------------------------------------- bf16 ----------

def test_bf16_hand_worked_patterns():
    vals = [1.0, -2.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -8 + 2.0 ** -30,
            3.0, 0.0, 2.0 ** -130, 65280.0]
    expect = [0x3F80, 0xC000, 0x3F80, 0x3F82, 0x3F81, 0x4040, 0x0000, 0x0008, 0x477F]
    assert list(bf16.encode(np.array(vals))) == expect


def test_bf16_decode_roundtrip_all_finite_patterns():
    bits = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    v = bf16.decode(bits)
    fin = np.isfinite(v)
    back = bf16.encode(v[fin])
    # +0 / -0 keep their sign bit
    assert np.array_equal(back, bits[fin])


def test_bf16_rne_matches_torch_from_binary32():
    """For binary32 inputs one-step rounding equals torch's float32 -> bfloat16 cast."""
    x = (_rng(8).standard_normal(200000) * np.exp(_rng(9).uniform(-20, 20, 200000))).astype(np.float32)
    # include exact ties: 9-bit odd significands sit half-way between two bf16 values
    odd = np.arange(128, 256, dtype=np.float32) * 2 + 1
    ties = np.concatenate([odd * np.float32(2.0 ** e) for e in (-9, -20, 3, 40)])
    x = np.concatenate([x, ties, -ties])
    expect = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = bf16.encode(x.astype(np.float64))
    assert np.array_equal(got, expect)


def test_bf16_overflow_rounds_to_signed_infinity():
    big = 3.3895313892515355e38                      # the largest finite bf16, 0x7F7F
    vals = np.array([big, -big, 3.39e38, -3.39e38, 1e39, -1e39, 3.3962e38, -3.3962e38])   # midpoint 3.39618e38
    assert bf16.encode(vals).tolist() == [0x7F7F, 0xFF7F, 0x7F7F, 0xFF7F, 0x7F80, 0xFF80, 0x7F80, 0xFF80]
    assert bf16.round_to_bf16_value(vals).tolist() == [big, -big, big, -big, np.inf, -np.inf, np.inf, -np.inf]
    # binary32 values near the top of the range, both signs, against torch's cast
    x = np.linspace(3.3e38, 3.4028234e38, 4001).astype(np.float32)
    x = np.concatenate([x, -x])
    expect = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(bf16.encode(x.astype(np.float64)), expect)


def test_bf16_rne_matches_torch_across_the_subnormal_boundary():
    """Every binary32 value on a 2^-140 grid from 2^-135 to 2^-124: bf16's subnormal
    quantum 2^-133 below 2^-126, its 8-bit significand above (including the band just
    under the smallest normal, where the two quanta differ)."""
    k = np.arange(2 ** 5, 2 ** 16 + 1, dtype=np.float64)
    x = (k * 2.0 ** -140).astype(np.float32)
    x = np.concatenate([x, -x])
    expect = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(bf16.encode(x.astype(np.float64)), expect)


# ---- Llama-3 frequency scaling ------------------------------------------------------

LLAMA31 = rope.Llama3Scaling(8.0, 1.0, 4.0, 8192.0)


def test_llama3_scaling_hand_values():
    """Worked by hand from the definition (P = 8192, low 1, high 4, factor 8): a wavelength
    of 4096 sits between P/4 = 2048 and P/1 = 8192 with blend weight (8192/4096 - 1) / 3 =
    1/3, so omega' = (2/3)(omega/8) + (1/3) omega = (5/12) omega; wavelength 1000 < 2048
    keeps omega; wavelength 10000 > 8192 gives omega / 8."""
    w = 2 * np.pi / np.array([4096.0, 1000.0, 10000.0])
    got = rope.llama3_scale(w, LLAMA31)
    assert np.allclose(got / w, [5.0 / 12.0, 1.0, 0.125], rtol=1e-14, atol=0)


def test_llama3_scaling_is_continuous_and_monotone_at_the_edges():
    P = LLAMA31.original_max_position
    for lam in (P / LLAMA31.high_freq_factor, P / LLAMA31.low_freq_factor):
        w = 2 * np.pi / np.array([lam * (1 - 1e-12), lam, lam * (1 + 1e-12)])
        g = rope.llama3_scale(w, LLAMA31)
        assert np.allclose(g, g[1], rtol=1e-9, atol=0)
    lam = np.geomspace(10, 1e7, 4001)
    g = rope.llama3_scale(2 * np.pi / lam, LLAMA31)
    assert np.all(np.diff(g) < 0)                 # still strictly decreasing in wavelength


def test_llama3_scaling_identity_and_inv_freq_plumbing():
    w = rope.inv_freq(5e5, 128)
    assert np.allclose(rope.llama3_scale(w, rope.Llama3Scaling(1.0, 1.0, 4.0, 8192.0)), w, rtol=1e-15, atol=0)
    spec = rope.RopeSpec(5e5, LLAMA31)
    ws = rope.inv_freq(spec, 128)
    assert ws[0] == w[0] == 1.0                   # the fastest pair keeps its frequency
    assert ws[-1] == w[-1] / 8.0                  # the slowest is divided by the factor
    x = np.random.default_rng(1).standard_normal((3, 128))
    pos = np.array([0, 5000, 123456])
    y = rope.rotate(x, pos, spec)
    assert np.allclose(rope.rotate(y, pos, spec, inverse=True), x, atol=1e-12)
    assert np.allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), atol=1e-12)


# ---- Hugging Face numerics ------------------------------------------------------------

def test_hf_rotation_worked_example():
    """Worked by hand: pair i = 0 has omega = 1, so at t = 1 the fp32 angle is 1 rad;
    cos 1 = 0.54030... = 1.0806 x 2^-1 rounds to 138/128 x 2^-1 = 0.5390625 in bf16 and
    sin 1 = 0.84147... = 1.6829 x 2^-1 to 215/128 x 2^-1 = 0.83984375.  For (a, b) = (1, 1):
    a' = r(0.5390625 - 0.83984375) = -0.30078125 (exact), b' = r(0.5390625 + 0.83984375) =
    r(1.37890625) = 1.375 (176.5/128 is a tie, rounded to even).  For (1, 0): (c, s)."""
    x = np.zeros((2, 128))
    x[0, 0], x[0, 64] = 1.0, 1.0
    x[1, 0] = 1.0
    y = rope.rotate_hf(x, np.array([1, 1]), 1e6)
    assert y[0, 0] == -0.30078125 and y[0, 64] == 1.375
    assert y[1, 0] == 0.5390625 and y[1, 64] == 0.83984375
    c, s = rope.hf_cos_sin(np.array([1]), 1e6, 128)
    assert c[0, 0] == 0.5390625 and s[0, 0] == 0.83984375


def test_hf_angles_are_torch_binary32_products():
    """The Hugging Face forward forms the angle as a binary32 product of binary32(t) and
    binary32(omega_i): computed here with torch in float32 (positions past 2^24 included,
    where binary32(t) is itself rounded), then cos / sin in float64."""
    d, theta = 128, 1e6
    t = np.array([0, 1, 77, 30001, 2 ** 20 + 3, 2 ** 24 + 1, 2 ** 25 + 3, 123456789])
    w32 = torch.from_numpy(rope.inv_freq(theta, d).astype(np.float32))
    ang = (torch.from_numpy(t.astype(np.float32))[:, None] * w32[None, :]).double().numpy()
    c, s = rope.hf_cos_sin(t, theta, d, bf16_cache=False)
    assert np.array_equal(c, np.cos(ang).astype(np.float32).astype(np.float64))
    assert np.array_equal(s, np.sin(ang).astype(np.float32).astype(np.float64))
    cb, sb = rope.hf_cos_sin(t, theta, d)
    assert np.array_equal(cb, bf16.round_to_bf16_value(np.cos(ang)))
    assert np.array_equal(sb, bf16.round_to_bf16_value(np.sin(ang)))
    # an fp64 angle would differ: the check above sees the binary32 rounding points
    assert not np.array_equal(c, np.cos(np.outer(t, rope.inv_freq(theta, d))).astype(np.float32))


def test_hf_rotation_with_a_binary32_cache_returns_binary32_values():
    x = _rng(31).standard_normal((5, 64))
    y = rope.rotate_hf(x, np.arange(5) * 1000, 1e4, bf16_cache=False)
    assert np.array_equal(y, y.astype(np.float32).astype(np.float64))
    assert not np.array_equal(y, bf16.round_to_bf16_value(y))


def test_hf_rotation_properties():
    """Position 0 is the identity (cos 1, sin 0 exactly); results are bf16 values; the HF
    rotation stays within the bf16 rounding of the exact one; its inverse undoes it up to
    that rounding."""
    rng = np.random.default_rng(4)
    from oracle import bf16
    x = bf16.round_to_bf16_value(rng.standard_normal((16, 128)))
    assert np.array_equal(rope.rotate_hf(x, np.zeros(16, dtype=int), 5e5), x)
    pos = rng.integers(0, 40000, size=16)
    y = rope.rotate_hf(x, pos, 5e5)
    assert np.array_equal(y, bf16.round_to_bf16_value(y))
    ex = rope.rotate(x, pos, 5e5)
    mag = np.concatenate([np.abs(x[:, :64]) + np.abs(x[:, 64:])] * 2, axis=-1)
    assert np.all(np.abs(y - ex) <= 2.0 ** -6 * mag + 1e-6 * np.abs(pos)[:, None] * mag)
    back = rope.rotate_hf(y, pos, 5e5, inverse=True)
    assert np.all(np.abs(back - x) <= 2.0 ** -5 * mag + 1e-6 * np.abs(pos)[:, None] * mag)
