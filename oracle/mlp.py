"""Applying the MLP mapper (oracle; test infrastructure only).

Sec. 4.3 ("Substituting MLP for ridge") and Appendix "Run information" (MLP baseline
architecture): per (target layer l, head h, K|V) the ridge map X W + b is replaced by
    y = Linear(hidden, d)( ReLU( Linear(hidden, hidden)( ReLU( Linear(d_s, hidden)(x) ) ) ) )
with hidden = 1024 in the paper, on the same source feature as the ridge mapper: the k
selected source layers' KV heads concatenated (cross-head, d_s = k n_kv d, keys with the
source RoPE stripped), and the same output handling (keys re-rotated with the target RoPE
after the bias, Sec. 3.3).  Only applying the MLP is covered; training it is not.

Linear layers use the nn.Linear convention: weight [out][in], Linear(z) = z W^T + b.

Rounding models:
* ``"exact"``   -- float64 throughout.
* ``"bf16fwd"`` -- a bf16 forward (Appendix "Run information"): the stripped source keys
                   are rounded to bf16 before the first layer (as in the ridge oracle) and
                   each hidden activation is rounded to bf16 after its ReLU (the tensors a
                   bf16 forward stores); the products and sums between those points, the
                   bias and the re-rotation are exact.  (Reading: the paper says only
                   "bfloat16 (forward)"; these are the points where such a forward holds
                   bf16 tensors.)
"""
import numpy as np

from . import bf16, rope


def mlp_forward(X, W1, b1, W2, b2, W3, b3, round_hidden=False):
    """Three-layer ReLU MLP on the rows of X [N][d_s] -> [N][d_out], float64.

    ``round_hidden``: round each hidden activation (after its ReLU) to bf16."""
    X = np.asarray(X, dtype=np.float64)
    h = np.maximum(X @ np.asarray(W1, dtype=np.float64).T + np.asarray(b1, dtype=np.float64), 0.0)
    if round_hidden:
        h = bf16.round_to_bf16_value(h)
    h = np.maximum(h @ np.asarray(W2, dtype=np.float64).T + np.asarray(b2, dtype=np.float64), 0.0)
    if round_hidden:
        h = bf16.round_to_bf16_value(h)
    return h @ np.asarray(W3, dtype=np.float64).T + np.asarray(b3, dtype=np.float64)


def cross_head_features(src, l, sel, kv, positions, theta_s, mode="exact", rope_numerics="exact"):
    """Source feature of target layer l: src [L_s][H][N][d] (one of K / V), the k layers
    sel[l] in order, each with all H heads (head-minor): [N][k H d].  Keys are stripped
    (and rounded to bf16 in ``"bf16fwd"`` mode; ``rope_numerics="hf"``: the Hugging Face
    forward's strip, rope.rotate_hf)."""
    parts = []
    for j in sel[l]:
        x = np.asarray(src[j], dtype=np.float64)            # [H][N][d]
        if kv == 0 and rope_numerics == "hf":
            x = rope.rotate_hf(x, np.asarray(positions)[None, :], theta_s, inverse=True)
        elif kv == 0:
            x = rope.rotate(x, np.asarray(positions)[None, :], theta_s, inverse=True)
            if mode == "bf16fwd":
                x = bf16.round_to_bf16_value(x)
        parts.append(np.concatenate(list(x), axis=-1))      # [N][H d], head-minor
    return np.concatenate(parts, axis=-1)


def map_tokens_mlp(src_k, src_v, positions, sel, params, theta_s, theta_t, mode="exact", rope_numerics="exact"):
    """src_k / src_v [L_s][H][N][d], positions [N], sel [L_t][k];
    params: W1 [L_t][2][H][hidden][k H d], b1 [L_t][2][H][hidden], W2 [L_t][2][H][hidden][hidden],
    b2 [L_t][2][H][hidden], W3 [L_t][2][H][d][hidden], b3 [L_t][2][H][d].
    Returns (out_k, out_v), each [L_t][H][N][d] float64 (keys re-rotated with theta_t)."""
    W1, b1, W2, b2, W3, b3 = (params[n] for n in ("W1", "b1", "W2", "b2", "W3", "b3"))
    Lt = len(sel)
    H = np.asarray(src_k).shape[1]
    outs = []
    for kv, src in enumerate((src_k, src_v)):
        out = []
        for l in range(Lt):
            X = cross_head_features(src, l, sel, kv, positions, theta_s, mode, rope_numerics)
            heads = []
            for h in range(H):
                y = mlp_forward(X, W1[l][kv][h], b1[l][kv][h], W2[l][kv][h], b2[l][kv][h], W3[l][kv][h],
                                b3[l][kv][h], round_hidden=(mode == "bf16fwd"))
                if kv == 0 and rope_numerics == "hf":
                    y = rope.rotate_hf(y, np.asarray(positions), theta_t)
                elif kv == 0:
                    y = rope.rotate(y, np.asarray(positions), theta_t)
                heads.append(y)
            out.append(np.stack(heads))
        outs.append(np.stack(out))
    return outs[0], outs[1]
