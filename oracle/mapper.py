"""Applying the fitted cross-model KV mapper (oracle; test infrastructure only).

What is computed, for target layer l, K/V, head h and every token with absolute
position t (the same t in source and target, Sec. 3.3):

1. x_j = source cache of layer sel[l][j], head h, token t, for j = 0..k-1
   (the top-k selected source layers, ascending; Sec. 3.2).
2. Keys only: x_j <- R_{Theta_s}(t)^{-1} x_j  (strip the source RoPE; Sec. 3.3).
3. X = [x_0 || ... || x_{k-1}]  (cross-layer concatenation, Sec. 3.2).
4. y = X W^{l,h} + b^{l,h}  (Eq. ridge_kv, row-vector convention of Sec. 2.3).
5. Keys only: y <- R_{Theta_t}(t) y  (re-apply the target RoPE; the composition
   K_t = (K_s R_s^{-1}(t) W_K + b_K) R_t(t) of Sec. 3.3: the bias is inside the
   rotated bracket).  Values are never rotated.

Two feature layouts:
* ``"per_head"``   -- x_j is head h of layer sel[l][j] only: F = k d.
* ``"cross_head"`` -- x_j is all KV heads of layer sel[l][j], head-minor
                      (the paper's d_s = k n_kv d; Sec. 3.1, Sec. 3.2, Appendix
                      "Run information", source-feature row): F = k H d.
The per-head map equals the cross-head map with W zero outside head h's rows.

RoPE numerics (``rope_numerics``): ``"exact"`` (the definition above) or ``"hf"`` -- the
rounding of the Hugging Face forward that wrote the caches (rope.rotate_hf: fp32 angle,
cos / sin and every product and sum of the rotation rounded to the cache dtype, the mapped
key rounded before the target rotation).

Two rounding models:
* ``"exact"``   -- everything in float64.
* ``"bf16fwd"`` -- the paper's forward runs in bf16 (Appendix "Run information"):
                   the stripped keys are materialised in bf16 (round-to-nearest-even)
                   before the contraction.  Values are already bf16 inputs, and the
                   contraction, bias and re-rotation stay exact.  This is the one point
                   where a bf16 forward rounds an operand of the contraction.

Rounding slack (bf16fwd only).  Rounding a stripped key to bf16 is a decision taken
on a value that any implementation computes with some error.  When the exact value
lies within that error of a bf16 rounding midpoint, both neighbours are correct
bf16-forward results.  ``map_tokens(..., rounding_slack=delta)`` therefore also
returns, for every output, the largest change that choosing the other neighbour for
every such ambiguous key element can cause: sum_f (hi_f - lo_f) |W[f][c]|, where
lo_f, hi_f are the roundings of x_f -/+ delta (|a| + |b|) (a, b the stored pair of
x_f), and for keys the two members of each re-rotated pair add up.  Values carry no
such decision, so their slack is zero.
"""
import numpy as np

from . import bf16, rope


def _pair_magnitude(x, style):
    """|a| + |b| of the RoPE pair each element belongs to (same shape as x)."""
    d = x.shape[-1]
    if style == "half":
        m = np.abs(x[..., : d // 2]) + np.abs(x[..., d // 2:])
        return np.concatenate([m, m], axis=-1)
    m = np.abs(x[..., 0::2]) + np.abs(x[..., 1::2])
    out = np.empty_like(x)
    out[..., 0::2] = m
    out[..., 1::2] = m
    return out


def _pair_sum(y, style):
    """Each element replaced by the sum over its RoPE pair (bound after a rotation)."""
    d = y.shape[-1]
    if style == "half":
        m = y[..., : d // 2] + y[..., d // 2:]
        return np.concatenate([m, m], axis=-1)
    m = y[..., 0::2] + y[..., 1::2]
    out = np.empty_like(y)
    out[..., 0::2] = m
    out[..., 1::2] = m
    return out


def map_tokens(src_k, src_v, positions, sel, W, b, theta_s, theta_t,
               mode="exact", style="half", head_mix="per_head", rounding_slack=None,
               rope_numerics="exact"):
    """Map a set of tokens.

    src_k, src_v : float64 [L_s][H][N][d]  -- stored (rotated) source keys, values.
    positions    : int [N]                 -- absolute positions of the N tokens.
    sel          : int [L_t][k]            -- selected source layers, ascending.
    W            : float64 [L_t][2][H][F][d]  (index 0 = K, 1 = V).
    b            : float64 [L_t][2][H][d] or None (zero bias).
    Returns (out_k, out_v), float64 [L_t][H][N][d]; with ``rounding_slack`` (bf16fwd
    mode) also (slack_k, slack_v) of the same shape.
    """
    src_k = np.asarray(src_k, dtype=np.float64)
    src_v = np.asarray(src_v, dtype=np.float64)
    pos = np.asarray(positions)
    sel = np.asarray(sel)
    Ls, H, N, d = src_k.shape
    Lt, k = sel.shape
    hf = rope_numerics == "hf"
    if hf:   # the HF forward's strip: already rounded to bf16 (mode bf16fwd)
        stripped = rope.rotate_hf(src_k, pos[None, None, :], theta_s, inverse=True, style=style,
                                  bf16_cache=(mode == "bf16fwd"))
    else:
        stripped = rope.rotate(src_k, pos[None, None, :], theta_s, inverse=True, style=style)
    feats = (stripped, src_v)
    out = np.empty((2, Lt, H, N, d), dtype=np.float64)
    want_slack = rounding_slack is not None and mode == "bf16fwd"
    slack = np.zeros_like(out) if rounding_slack is not None else None
    if want_slack:
        delta = rounding_slack * _pair_magnitude(src_k, style)
        amb = (bf16.round_to_bf16_value(stripped + delta) -
               bf16.round_to_bf16_value(stripped - delta))
    for l in range(Lt):
        for kv in range(2):
            for h in range(H):
                if head_mix == "per_head":
                    parts = [feats[kv][s, h] for s in sel[l]]
                elif head_mix == "cross_head":
                    parts = [feats[kv][s, hh] for s in sel[l] for hh in range(H)]
                else:
                    raise ValueError(head_mix)
                X = np.concatenate(parts, axis=-1)
                if mode == "bf16fwd" and kv == 0:
                    X = bf16.round_to_bf16_value(X)
                elif mode not in ("exact", "bf16fwd"):
                    raise ValueError(mode)
                Y = X @ W[l, kv, h]
                if b is not None:
                    Y = Y + b[l, kv, h]
                if kv == 0:
                    Y = (rope.rotate_hf(Y, pos, theta_t, style=style, bf16_cache=(mode == "bf16fwd")) if hf
                         else rope.rotate(Y, pos, theta_t, style=style))
                out[kv, l, h] = Y
                if want_slack and kv == 0:
                    if head_mix == "per_head":
                        A = np.concatenate([amb[s, h] for s in sel[l]], axis=-1)
                    else:
                        A = np.concatenate([amb[s, hh] for s in sel[l] for hh in range(H)], axis=-1)
                    slack[0, l, h] = _pair_sum(A @ np.abs(W[l, 0, h]), style)
    if rounding_slack is not None:
        return out[0], out[1], slack[0], slack[1]
    return out[0], out[1]


def map_cache(src_k, src_v, positions, sel, W, b, theta_s, theta_t,
              mode="exact", style="half", head_mix="per_head", rounding_slack=None,
              rope_numerics="exact"):
    """Contiguous-cache form: src [L_s][B][H][T][d], positions [B][T] ->
    (out_k, out_v) [L_t][B][H][T][d] (plus the two slacks with ``rounding_slack``)."""
    src_k = np.asarray(src_k, dtype=np.float64)
    src_v = np.asarray(src_v, dtype=np.float64)
    Ls, B, H, T, d = src_k.shape
    pos = np.asarray(positions).reshape(B * T)

    def tok(x):  # [L][B][H][T][d] -> [L][H][B*T][d]
        return x.transpose(0, 2, 1, 3, 4).reshape(x.shape[0], H, B * T, d)

    res = map_tokens(tok(src_k), tok(src_v), pos, sel, W, b, theta_s, theta_t,
                     mode, style, head_mix, rounding_slack, rope_numerics)
    Lt = res[0].shape[0]

    def untok(y):
        return y.reshape(Lt, H, B, T, d).transpose(0, 2, 1, 3, 4)

    return tuple(untok(r) for r in res)


def mapper_params(L_t, n_kv_t, d_t, k, n_kv_s=None, d_s=None, head_mix="cross_head"):
    """Mapper size, K plus V (Appendix C, serving cost):
    cross-head  2 L_t n_kv^t (k n_kv^s d_h^s) d_h^t;  per-head  2 L_t n_kv^t (k d_h^s) d_h^t."""
    n_kv_s = n_kv_t if n_kv_s is None else n_kv_s
    d_s = d_t if d_s is None else d_s
    feat = k * n_kv_s * d_s if head_mix == "cross_head" else k * d_s
    return 2 * L_t * n_kv_t * feat * d_t
