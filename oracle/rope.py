"""RoPE rotation R_Theta(t) and its inverse (oracle; test infrastructure only).

Sec. 3.3 (content-space mapping): the cache stores rotated keys
k_RoPE(t) = R_Theta(t) k_content; the inverse R_Theta(t)^{-1} = R_Theta(-t) strips
the rotation exactly because R is orthogonal.

Standard RoPE (Su et al., cited in Sec. 3.3) rotates channel pair i by the angle
t * omega_i with omega_i = theta^(-2i/d), i = 0 .. d/2-1, as the complex product
(a + i b) * exp(i t omega_i), i.e.  a' = a cos - b sin,  b' = a sin + b cos.

Pair layout (the paper does not state one):
* ``"half"``        -- pairs (i, i + d/2): the layout of the Qwen3 / Llama checkpoints.
* ``"interleaved"`` -- pairs (2i, 2i+1).

Frequency scaling.  The Llama 3.1 checkpoints of the paper's Llama pairs rescale the
inverse frequencies ("llama3" rope scaling, published with those checkpoints; the paper
itself does not discuss it).  ``theta`` may be a plain base or a ``RopeSpec`` carrying such
a scaling; every function here accepts either.
"""
from typing import NamedTuple, Optional

import numpy as np


class Llama3Scaling(NamedTuple):
    factor: float                   # long wavelengths are divided by this
    low_freq_factor: float
    high_freq_factor: float
    original_max_position: float    # context length the model was pre-trained with


class RopeSpec(NamedTuple):
    theta: float
    scaling: Optional[Llama3Scaling] = None


def llama3_scale(omega, s):
    """Scaled inverse frequencies: with wavelength lam = 2 pi / omega, keep omega where
    lam < P / high_freq_factor, divide by factor where lam > P / low_freq_factor, and in
    between blend (1 - a) omega / factor + a omega with a = (P / lam - low_freq_factor) /
    (high_freq_factor - low_freq_factor); P = original_max_position."""
    omega = np.asarray(omega, dtype=np.float64)
    lam = 2.0 * np.pi / omega
    P = float(s.original_max_position)
    a = (P / lam - s.low_freq_factor) / (s.high_freq_factor - s.low_freq_factor)
    blend = (1.0 - a) * omega / s.factor + a * omega
    out = np.where(lam < P / s.high_freq_factor, omega, blend)
    return np.where(lam > P / s.low_freq_factor, omega / s.factor, out)


def inv_freq(theta, d):
    """omega_i = theta^(-2i/d) for i in [0, d/2), float64 (scaled when ``theta`` is a
    RopeSpec with a scaling)."""
    spec = theta if isinstance(theta, RopeSpec) else RopeSpec(float(theta))
    i = np.arange(d // 2, dtype=np.float64)
    omega = np.power(np.float64(spec.theta), -2.0 * i / d)
    return omega if spec.scaling is None else llama3_scale(omega, spec.scaling)


def angles(positions, theta, d):
    """t * omega_i in float64; shape positions.shape + (d/2,)."""
    p = np.asarray(positions, dtype=np.float64)
    return p[..., None] * inv_freq(theta, d)


def _pairs(x, style):
    d = x.shape[-1]
    if style == "half":
        return x[..., : d // 2], x[..., d // 2:]
    if style == "interleaved":
        return x[..., 0::2], x[..., 1::2]
    raise ValueError(style)


def _unpairs(a, b, style):
    if style == "half":
        return np.concatenate([a, b], axis=-1)
    out = np.empty(a.shape[:-1] + (2 * a.shape[-1],), dtype=np.float64)
    out[..., 0::2] = a
    out[..., 1::2] = b
    return out


def hf_cos_sin(positions, theta, d, bf16_cache=True):
    """cos and sin as the Hugging Face bf16 forward forms them: the angle is the fp32
    product of fp32(t) and fp32(omega_i) (omega_i rounded once from its exact value), its
    cos and sin are taken exactly and rounded to the cache dtype (bf16, or fp32)."""
    from . import bf16 as _bf16
    w32 = inv_freq(theta, d).astype(np.float32)
    p32 = np.asarray(positions).astype(np.float32)
    ang = (p32[..., None] * w32).astype(np.float32).astype(np.float64)   # fp32 multiply, rounded
    c, s = np.cos(ang), np.sin(ang)
    if bf16_cache:
        return _bf16.round_to_bf16_value(c), _bf16.round_to_bf16_value(s)
    return c.astype(np.float32).astype(np.float64), s.astype(np.float32).astype(np.float64)


def rotate_hf(x, positions, theta, inverse=False, style="half", bf16_cache=True):
    """The rotation with the rounding of a Hugging Face forward in the cache dtype: with
    (c, s) from hf_cos_sin and r() the rounding to the cache dtype,
        a' = r(r(a c) - r(b s)),  b' = r(r(b c) + r(a s))      (inverse: s -> -s).
    x is taken as a cache-dtype tensor (rounded first)."""
    from . import bf16 as _bf16

    def r(v):
        v = np.asarray(v, dtype=np.float64)
        return _bf16.round_to_bf16_value(v) if bf16_cache else v.astype(np.float32).astype(np.float64)

    x = r(x)
    d = x.shape[-1]
    c, s = hf_cos_sin(np.broadcast_to(np.asarray(positions), x.shape[:-1]), theta, d, bf16_cache)
    if inverse:
        s = -s
    a, b = _pairs(x, style)
    return _unpairs(r(r(a * c) - r(b * s)), r(r(b * c) + r(a * s)), style)


def rotate(x, positions, theta, inverse=False, style="half"):
    """Apply R_Theta(t) (or its inverse) to the last axis of ``x``.

    ``x``: float64 [..., d]; ``positions``: integer array broadcastable to x.shape[:-1].
    ``inverse=True`` applies R_Theta(t)^{-1} = R_Theta(-t) (the RoPE strip of Sec. 3.3).
    """
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    ang = angles(np.broadcast_to(np.asarray(positions), x.shape[:-1]), theta, d)
    if inverse:
        ang = -ang
    c, s = np.cos(ang), np.sin(ang)
    a, b = _pairs(x, style)
    return _unpairs(a * c - b * s, a * s + b * c, style)
