"""Pins for oracle.mlp (CPU): the MLP mapper of Sec. 4.3 / Appendix "Run information".

* A worked example with literal numbers (ReLU clipping, layer order, nn.Linear orientation).
* The ReLU identity relu(z) - relu(-z) = z turns a hidden layer of [A; -A] followed by
  [I, -I] into the linear map z A^T: the MLP then equals the (separately pinned) ridge
  mapper oracle.mapper.map_tokens in cross-head mode, keys stripped, bias inside the
  re-rotation.  A dropped term, a transposed weight, a wrong head or layer order or a
  rotation in the wrong place breaks it.
* A dead ReLU layer leaves only the last bias (rotated for keys).
* bf16fwd mode rounds the hidden activations to bf16 values."""
import numpy as np

from oracle import bf16, mapper, mlp, rope


def test_worked_example():
    # x = (1, -2); layer 1 (2 -> 3): pre-activations (1 - 2 + 0.5, 2*1 + 0, -1 - 1*(-2) - 3)
    x = np.array([[1.0, -2.0]])
    W1 = np.array([[1.0, 1.0], [2.0, 0.0], [-1.0, -1.0]])
    b1 = np.array([0.5, 0.0, -3.0])          # pre: (-0.5, 2, -2) -> relu (0, 2, 0)
    W2 = np.array([[1.0, 1.0, 1.0], [0.0, -1.0, 0.0]])
    b2 = np.array([1.0, 5.0])                # pre: (3, 3) -> relu (3, 3)
    W3 = np.array([[2.0, -1.0]])
    b3 = np.array([0.25])                    # 6 - 3 + 0.25
    y = mlp.mlp_forward(x, W1, b1, W2, b2, W3, b3)
    assert y.shape == (1, 1) and y[0, 0] == 3.25
    b2n = np.array([1.0, -5.0])              # second unit clipped: pre (3, -7) -> (3, 0)
    assert mlp.mlp_forward(x, W1, b1, W2, b2n, W3, b3)[0, 0] == 6.25


def _linear_as_mlp(Wlin, b, rng=None):
    """W_lin [F][d] (row-vector map x W + b) as MLP weights with hidden = 2d.

    z = x W_lin; layer 1 gives [relu(z + c); relu(-z - c)]; layer 2 scales both halves by
    a positive diagonal D and adds e1, e2 >= 0 (the ReLU is then inert); layer 3 takes
    D^-1 (first half - second half): relu(u) - relu(-u) = u leaves z + c + (e1 - e2) / D,
    and b3 = b - c - (e1 - e2) / D.  With ``rng`` every block gets its own c, D, e1, e2."""
    F, d = Wlin.shape
    if rng is None:
        c, D, e1, e2 = np.zeros(d), np.ones(d), np.zeros(d), np.zeros(d)
    else:
        c, D = rng.standard_normal(d), rng.uniform(0.5, 2.0, d)
        e1, e2 = rng.uniform(0.0, 1.0, d), rng.uniform(0.0, 1.0, d)
    W1 = np.concatenate([Wlin.T, -Wlin.T], axis=0)                      # [2d][F]
    W2 = np.diag(np.concatenate([D, D]))
    W3 = np.concatenate([np.diag(1.0 / D), -np.diag(1.0 / D)], axis=1)   # [d][2d]
    return W1, np.concatenate([c, -c]), W2, np.concatenate([e1, e2]), W3, b - c - (e1 - e2) / D


def test_relu_identity_reduces_to_the_ridge_mapper():
    rng = np.random.default_rng(5)
    Ls, Lt, H, N, d, k = 3, 2, 2, 9, 128, 2
    src_k = rng.standard_normal((Ls, H, N, d))
    src_v = rng.standard_normal((Ls, H, N, d))
    pos = rng.integers(0, 5000, size=N)
    sel = np.array([[0, 2], [1, 2]])
    F = k * H * d
    W = rng.standard_normal((Lt, 2, H, F, d)) / np.sqrt(F)
    b = rng.standard_normal((Lt, 2, H, d))
    params = {n: [] for n in ("W1", "b1", "W2", "b2", "W3", "b3")}
    for l in range(Lt):
        per_l = {n: [] for n in params}
        for kv in range(2):
            per_kv = {n: [] for n in params}
            for h in range(H):
                for n, v in zip(("W1", "b1", "W2", "b2", "W3", "b3"),
                                _linear_as_mlp(W[l, kv, h], b[l, kv, h], rng)):
                    per_kv[n].append(v)
            for n in params:
                per_l[n].append(per_kv[n])
        for n in params:
            params[n].append(per_l[n])
    params = {n: np.asarray(v) for n, v in params.items()}
    ok, ov = mlp.map_tokens_mlp(src_k, src_v, pos, sel, params, 1e6, 5e5)
    rk, rv = mapper.map_tokens(src_k, src_v, pos, sel, W, b, 1e6, 5e5, head_mix="cross_head")
    assert np.allclose(ok, rk, rtol=0, atol=1e-9) and np.allclose(ov, rv, rtol=0, atol=1e-9)
    # the Hugging Face rounding of the strip and the re-rotation (the MLP's HF forward
    # rounds both rotations to bf16, as the mapper's bf16 forward does): equal up to the
    # bf16 rounding of the output, whose pre-rounding values differ in the last f64 bits
    hk, hv = mlp.map_tokens_mlp(src_k, src_v, pos, sel, params, 1e6, 5e5, rope_numerics="hf")
    gk, gv = mapper.map_tokens(src_k, src_v, pos, sel, W, b, 1e6, 5e5, head_mix="cross_head",
                               mode="bf16fwd", rope_numerics="hf")
    assert np.all(np.abs(hk - gk) <= 2.0 ** -7 * np.abs(gk) + 1e-30)
    assert np.mean(hk == gk) > 0.99 and np.allclose(hv, rv, rtol=0, atol=1e-9)


def test_dead_relu_leaves_the_rotated_last_bias():
    rng = np.random.default_rng(6)
    Ls, Lt, H, N, d, k, hid = 2, 1, 1, 5, 128, 1, 16
    src_k = rng.standard_normal((Ls, H, N, d))
    src_v = rng.standard_normal((Ls, H, N, d))
    pos = np.arange(N) * 37
    sel = np.array([[1]])
    F = k * H * d
    b3 = rng.standard_normal((Lt, 2, H, d))
    params = dict(W1=rng.standard_normal((Lt, 2, H, hid, F)) * 0.01, b1=np.full((Lt, 2, H, hid), -1e3),
                  W2=rng.standard_normal((Lt, 2, H, hid, hid)), b2=np.zeros((Lt, 2, H, hid)),
                  W3=rng.standard_normal((Lt, 2, H, d, hid)), b3=b3)
    ok, ov = mlp.map_tokens_mlp(src_k, src_v, pos, sel, params, 1e6, 1e6)
    assert np.array_equal(ov[0, 0], np.broadcast_to(b3[0, 1, 0], (N, d)))
    want_k = rope.rotate(np.broadcast_to(b3[0, 0, 0], (N, d)), pos, 1e6)
    assert np.allclose(ok[0, 0], want_k, rtol=0, atol=1e-12)


def test_bf16fwd_rounds_hidden_activations():
    rng = np.random.default_rng(8)
    X = rng.standard_normal((7, 5))
    W1, b1 = rng.standard_normal((6, 5)), rng.standard_normal(6)
    W2, b2 = rng.standard_normal((6, 6)), rng.standard_normal(6)
    W3, b3 = rng.standard_normal((2, 6)), np.zeros(2)
    # with W3 = identity rows the output exposes the second hidden activation
    W3e = np.eye(6)
    h2 = mlp.mlp_forward(X, W1, b1, W2, b2, W3e, np.zeros(6), round_hidden=True)
    assert np.array_equal(h2, bf16.round_to_bf16_value(h2))
    exact = mlp.mlp_forward(X, W1, b1, W2, b2, W3, b3)
    rounded = mlp.mlp_forward(X, W1, b1, W2, b2, W3, b3, round_hidden=True)
    assert not np.array_equal(exact, rounded)
    assert np.allclose(exact, rounded, rtol=0.05, atol=0.05)


def test_bf16fwd_features_match_the_mapper_exactly():
    """bf16fwd rounds the stripped keys before the first layer, as the mapper does.  With
    one power-of-two entry per column of W_lin, and D a power of two, every hidden value
    is a scaled copy of one rounded feature, so the hidden roundings change nothing and
    the MLP equals the mapper's bf16 forward bit for bit."""
    rng = np.random.default_rng(9)
    Ls, Lt, H, N, d, k = 3, 2, 2, 5, 16, 2
    src_k = bf16.round_to_bf16_value(rng.standard_normal((Ls, H, N, d)))
    src_v = bf16.round_to_bf16_value(rng.standard_normal((Ls, H, N, d)))
    pos = np.array([0, 3, 700, 9000, 31111])
    sel = np.array([[0, 2], [1, 2]])
    F = k * H * d
    W = np.zeros((Lt, 2, H, F, d))
    b = rng.standard_normal((Lt, 2, H, d))
    params = {n: np.zeros((Lt, 2, H) + shp) for n, shp in
              (("W1", (2 * d, F)), ("b1", (2 * d,)), ("W2", (2 * d, 2 * d)), ("b2", (2 * d,)),
               ("W3", (d, 2 * d)), ("b3", (d,)))}
    for l in range(Lt):
        for kv in range(2):
            for h in range(H):
                rows = rng.integers(0, F, d)
                W[l, kv, h, rows, np.arange(d)] = rng.choice([-1.0, 1.0], d) * 2.0 ** rng.integers(-2, 3, d)
                D = 2.0 ** rng.integers(-2, 3, d)
                params["W1"][l, kv, h] = np.concatenate([W[l, kv, h].T, -W[l, kv, h].T])
                params["W2"][l, kv, h] = np.diag(np.concatenate([D, D]))
                params["W3"][l, kv, h] = np.concatenate([np.diag(1.0 / D), -np.diag(1.0 / D)], axis=1)
                params["b3"][l, kv, h] = b[l, kv, h]
    ok, ov = mlp.map_tokens_mlp(src_k, src_v, pos, sel, params, 1e4, 1e6, mode="bf16fwd")
    rk, rv = mapper.map_tokens(src_k, src_v, pos, sel, W, b, 1e4, 1e6, head_mix="cross_head", mode="bf16fwd")
    assert np.array_equal(ok, rk) and np.array_equal(ov, rv)
    ek, _ = mapper.map_tokens(src_k, src_v, pos, sel, W, b, 1e4, 1e6, head_mix="cross_head")
    assert not np.array_equal(ok, ek)


def test_bf16fwd_rounds_hidden_activations_inside_the_map():
    # W2 = W3 = I and zero later biases: the mapped values are the second hidden layer
    rng = np.random.default_rng(10)
    Ls, Lt, H, N, d, k = 2, 1, 1, 6, 8, 1
    src_k = rng.standard_normal((Ls, H, N, d))
    src_v = rng.standard_normal((Ls, H, N, d))
    F = k * H * d
    params = dict(W1=rng.standard_normal((Lt, 2, H, d, F)), b1=np.full((Lt, 2, H, d), 5.0),
                  W2=np.broadcast_to(np.eye(d), (Lt, 2, H, d, d)).copy(), b2=np.zeros((Lt, 2, H, d)),
                  W3=np.broadcast_to(np.eye(d), (Lt, 2, H, d, d)).copy(), b3=np.zeros((Lt, 2, H, d)))
    sel = np.array([[1]])
    _, v16 = mlp.map_tokens_mlp(src_k, src_v, np.arange(N), sel, params, 1e4, 1e4, mode="bf16fwd")
    _, v64 = mlp.map_tokens_mlp(src_k, src_v, np.arange(N), sel, params, 1e4, 1e4)
    assert np.array_equal(v16, bf16.round_to_bf16_value(v16)) and not np.array_equal(v64, v16)
    assert np.allclose(v16, v64, rtol=2.0 ** -7, atol=0)


def test_bf16fwd_rounds_the_stripped_keys_before_the_first_layer():
    """A first-layer unit that adds two stripped key channels: in bf16fwd the MLP sees
    bf16(s_0) + bf16(s_1) (the operand rounding of the bf16 forward), and its hidden
    rounding then gives bf16(bf16(s_0) + bf16(s_1)); rounding only after the sum would give
    bf16(s_0 + s_1), which differs for some tokens.  Brute force per token from the
    pinned strip (rope.rotate) and rounding (bf16.round_to_bf16_value)."""
    rng = np.random.default_rng(12)
    N, d = 256, 8
    src_k = bf16.round_to_bf16_value(rng.standard_normal((1, 1, N, d)))
    src_v = bf16.round_to_bf16_value(rng.standard_normal((1, 1, N, d)))
    pos = rng.integers(1, 30000, N)
    sel = np.array([[0]])
    zero = lambda *shp: np.zeros((1, 2, 1) + shp)
    params = dict(W1=zero(2, d), b1=zero(2), W2=np.broadcast_to(np.eye(2), (1, 2, 1, 2, 2)).copy(),
                  b2=zero(2), W3=zero(d, 2), b3=zero(d))
    params["W1"][0, :, 0, 0, :2] = 1.0            # hidden 0: s_0 + s_1
    params["W1"][0, :, 0, 1, :2] = -1.0           # hidden 1: -(s_0 + s_1)
    params["W3"][0, :, 0, 0] = [1.0, -1.0]        # output channel 0: relu(z) - relu(-z) = z
    ok, _ = mlp.map_tokens_mlp(src_k, src_v, pos, sel, params, 1e4, 1e4, mode="bf16fwd")
    z = rope.rotate(ok[0, 0], pos, 1e4, inverse=True)[:, 0]      # undo the target rotation
    s = rope.rotate(src_k[0, 0], pos, 1e4, inverse=True)
    r = bf16.round_to_bf16_value
    want = r(r(s[:, 0]) + r(s[:, 1]))
    assert np.allclose(z, want, rtol=1e-12, atol=1e-300)
    assert np.any(r(s[:, 0] + s[:, 1]) != want)                     # the case tells them apart
