"""GPU parity of the MLP mapper apply (kvx_mlp_map, Sec. 4.3 / Appendix "Run information")
against the float64 oracle (oracle.mlp in bf16fwd mode), through the C ABI.

Bound (derived from the arithmetic, interval form).  The kernel takes three rounding
decisions the oracle also takes -- a stripped key to bf16, each hidden activation to bf16
after its ReLU, the output to bf16 -- on values it computes with an error the test bounds:
* stripped keys: fp32 strip with |angle error| < 1e-6 rad, so a key x of the stored pair
  (a, b) is known within 4e-6 (|a| + |b|); r0 = the distance between the bf16 roundings
  of x -/+ that (zero unless x is that close to a rounding midpoint);
* a pre-activation z = sum_i x_i w_i + b accumulated in fp32 over K terms: within
  dz = sum |w_i| r_i + 2 K u sum |x_i w_i| + u |z| (u = 2^-24; the 2 allows a truncating
  tensor-core accumulator) of the oracle's;
* the stored activation bf16(relu(z)) then lies between bf16(relu(z - dz)) and
  bf16(relu(z + dz)) (rounding and ReLU are monotone), which gives the next layer's r;
* the output y (after the target RoPE for keys: pair sums of dy plus 4e-6 + 4u of the pair
  magnitude) is stored as bf16: the kernel's value must lie in
  [bf16(y - dy), bf16(y + dy)].
A dropped bias, a transposed or misplaced weight block, a wrong head or layer order moves
outputs far outside these intervals."""
import numpy as np
import pytest
import torch

from oracle import bf16 as obf16
from oracle import mapper as omapper
from oracle import mlp as omlp
from oracle import rope as orope
from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu

U = 2.0 ** -24


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_03893_gb300 import build as kbuild
    kbuild.build()
    kvx.lib()
    torch.cuda.set_device(0)


def _dec(t):
    return obf16.decode(t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))


def _weights(w, hid, seed, dev):
    """Seeded synthetic MLP weights on the device (bf16 weights, fp32 biases), scaled so the
    activations stay O(1) through the ReLU layers."""
    g = torch.Generator(device=dev).manual_seed(seed)
    ds = w.k * w.H * w.d
    shape = (w.Lt, 2, w.H)

    def rnd(*s, scale, dtype):
        t = torch.randn(*s, generator=g, device=dev, dtype=dtype)
        return t.mul_(scale).contiguous()

    return dict(W1=rnd(*shape, hid, ds, scale=1.0 / np.sqrt(ds), dtype=torch.bfloat16),
                b1=rnd(*shape, hid, scale=0.1, dtype=torch.float32),
                W2=rnd(*shape, hid, hid, scale=np.sqrt(2.0 / hid), dtype=torch.bfloat16),
                b2=rnd(*shape, hid, scale=0.1, dtype=torch.float32),
                W3=rnd(*shape, w.d, hid, scale=np.sqrt(2.0 / hid), dtype=torch.bfloat16),
                b3=rnd(*shape, w.d, scale=0.1, dtype=torch.float32))


def _run(w, hid, sel, params, sk, sv, pos, workspace=None):
    dev = sk.device
    tk = torch.full((w.Lt, w.B, w.H, w.T, w.d), float("nan"), dtype=torch.bfloat16, device=dev)
    tv = torch.full_like(tk, float("nan"))
    posd = torch.from_numpy(pos).to(dev)
    ws_ptr, ws_bytes = (None, 0) if workspace is None else (workspace.data_ptr(), workspace.numel())
    cfg = kvx.mlp_config(w.Ls, w.Lt, w.H, w.d, w.k, hid, w.theta_s, w.theta_t, sel,
                         params["W1"].data_ptr(), params["b1"].data_ptr(), params["W2"].data_ptr(),
                         params["b2"].data_ptr(), params["W3"].data_ptr(), params["b3"].data_ptr(),
                         ws_ptr, ws_bytes)
    kvx.kvx_mlp_map(cfg, kvx.src_from_tensors(sk, sv), w.B, w.T, posd.data_ptr(), kvx.tgt_from_tensors(tk, tv),
                    torch.cuda.current_stream().cuda_stream)
    return tk, tv, cfg


def _layer(x, r, W, b):
    """fp32-accumulated pre-activation bound: (z, dz)."""
    z = x @ W.T + b
    dz = r @ np.abs(W).T + 2 * W.shape[1] * U * (np.abs(x) @ np.abs(W).T) + U * np.abs(z)
    return z, dz


def _act(z, dz):
    """bf16(relu(z)) and the distance to the roundings of relu(z -/+ dz)."""
    h = obf16.round_to_bf16_value(np.maximum(z, 0.0))
    lo = obf16.round_to_bf16_value(np.maximum(z - dz, 0.0))
    hi = obf16.round_to_bf16_value(np.maximum(z + dz, 0.0))
    return h, np.maximum(hi - h, h - lo)


def _check(w, hid, sel, P, src_tok, pos_flat, gpu_out, cases):
    """cases: (l, kv, h, token indices).  src_tok: dict kv -> [L_s][H][N][d] float64 stored."""
    worst = 0.0
    for (l, kv, h, toks) in cases:
        X = omlp.cross_head_features(src_tok[kv], l, sel, kv, pos_flat, w.theta_s, mode="bf16fwd")[toks]
        if kv == 0:
            parts = []
            for j in sel[l]:
                s = src_tok[0][j][:, toks]                                   # [H][n][d] stored
                st = orope.rotate(s, pos_flat[toks][None, :], w.theta_s, inverse=True)
                delta = 4e-6 * omapper._pair_magnitude(s, "half")
                amb = obf16.round_to_bf16_value(st + delta) - obf16.round_to_bf16_value(st - delta)
                parts.append(np.concatenate(list(amb), axis=-1))
            r0 = np.concatenate(parts, axis=-1)
        else:
            r0 = np.zeros_like(X)
        W1, b1 = _dec(P["W1"][l, kv, h]), P["b1"][l, kv, h].cpu().double().numpy()
        W2, b2 = _dec(P["W2"][l, kv, h]), P["b2"][l, kv, h].cpu().double().numpy()
        W3, b3 = _dec(P["W3"][l, kv, h]), P["b3"][l, kv, h].cpu().double().numpy()
        z1, dz1 = _layer(X, r0, W1, b1)
        h1, r1 = _act(z1, dz1)
        z2, dz2 = _layer(h1, r1, W2, b2)
        h2, r2 = _act(z2, dz2)
        y, dy = _layer(h2, r2, W3, b3)
        # the reference itself comes from the oracle
        ref = omlp.mlp_forward(X, W1, b1, W2, b2, W3, b3, round_hidden=True)
        assert np.allclose(ref, y, rtol=0, atol=1e-9)
        if kv == 0:
            mag = omapper._pair_magnitude(ref, "half")
            ref = orope.rotate(ref, pos_flat[toks], w.theta_t)
            dy = omapper._pair_sum(dy, "half") + mag * (4e-6 + 4 * U)
        lo = obf16.round_to_bf16_value(ref - dy)
        hi = obf16.round_to_bf16_value(ref + dy)
        b_idx, t_idx = toks // w.T, toks % w.T
        g = _dec(gpu_out[kv][l][:, h][torch.from_numpy(b_idx), torch.from_numpy(t_idx)])   # [n][d]
        inside = (g >= lo) & (g <= hi)
        assert inside.all(), "l=%d kv=%d h=%d: %d outside, max excess %.3g (ref %.4g gpu %.4g)" % (
            l, kv, h, (~inside).sum(), np.max(np.maximum(lo - g, g - hi)), ref[~inside][0], g[~inside][0])
        worst = max(worst, float(np.max(np.abs(g - ref) / np.maximum(dy + 2.0 ** -8 * np.abs(ref), 1e-30))))
        # the intervals are worst-case; typical outputs sit within the bf16 rounding of the
        # block's scale (2^-7 of its RMS; a systematic error such as a wrong bias or head
        # moves most of them further).  Not one step of each output's own magnitude: after
        # a cancellation (RoPE pair, final sum) an output is small and its error is not.
        rms = np.sqrt(np.mean(ref * ref))
        close = np.mean(np.abs(g - ref) <= 2.0 ** -7 * rms)
        assert close >= 0.99, "l=%d kv=%d h=%d: only %.4f of outputs within 2^-7 RMS" % (l, kv, h, close)
    return worst


def _tok(cache):
    x = _dec(cache)
    L, B, H, T, d = x.shape
    return x.transpose(0, 2, 1, 3, 4).reshape(L, H, B * T, d)


@pytest.mark.parametrize("over,hid", [
    (dict(Ls=3, Lt=2, H=2, B=2, T=300, k=2), 256),                   # B > 1, ragged token tiles
    (dict(Ls=4, Lt=3, H=2, B=1, T=200, k=3, theta_t=5e5), 1024),     # the paper's hidden width, two thetas
    (dict(Ls=2, Lt=2, H=4, B=1, T=64, k=1), 512),                    # one short tile, four heads
])
def test_mlp_small_every_output(over, hid):
    w = syn.workload("qwen3_14b_32b_b8x1024_k4_xhead", **over)
    dev = torch.device("cuda:0")
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    pos = syn.positions(w)
    P = _weights(w, hid, 11, dev)
    tk, tv, _ = _run(w, hid, sel, P, sk, sv, pos)
    assert not torch.isnan(tk.float()).any() and not torch.isnan(tv.float()).any(), "unwritten outputs"
    src_tok = {0: _tok(sk), 1: _tok(sv)}
    N = w.B * w.T
    cases = [(l, kv, h, np.arange(N)) for l in range(w.Lt) for kv in range(2) for h in range(w.H)]
    _check(w, hid, sel, P, src_tok, pos.reshape(-1), (tk, tv), cases)


def test_mlp_layer_groups_match_one_pass():
    """A caller workspace that holds one target layer's hidden activations (layer groups of
    one) gives the same bytes as a workspace that holds every layer at once."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4_xhead", Ls=3, Lt=3, H=2, B=1, T=256, k=2)
    dev = torch.device("cuda:0")
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    pos = syn.positions(w)
    P = _weights(w, 256, 12, dev)
    cfg = kvx.mlp_config(w.Ls, w.Lt, w.H, w.d, w.k, 256, w.theta_s, w.theta_t, sel, *(P[n].data_ptr() for n in
                         ("W1", "b1", "W2", "b2", "W3", "b3")))
    full = kvx.kvx_mlp_workspace_bytes(cfg, w.B, w.T)
    per_layer = 2 * 2 * w.B * w.T * w.H * 256 * 2
    a = _run(w, 256, sel, P, sk, sv, pos, torch.empty(full, dtype=torch.uint8, device=dev))
    b = _run(w, 256, sel, P, sk, sv, pos, torch.empty(full - 2 * per_layer, dtype=torch.uint8, device=dev))
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])
    with pytest.raises(kvx.KvxError) as e:
        _run(w, 256, sel, P, sk, sv, pos, torch.empty(4096, dtype=torch.uint8, device=dev))
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_mlp_headline_shapes_sampled():
    """Qwen3-14B -> 32B layer and head counts, k = 4 (d_s = 4096), hidden 1024, 384 tokens:
    every output on the GPU, sampled (layer, K|V, head) blocks of 48 tokens checked."""
    w = syn.workload("qwen3_14b_32b_t32768_k4_xhead", T=384)
    dev = torch.device("cuda:0")
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    pos = syn.positions(w)
    P = _weights(w, 1024, 13, dev)
    tk, tv, _ = _run(w, 1024, sel, P, sk, sv, pos)
    assert not torch.isnan(tk.float()).any() and not torch.isnan(tv.float()).any()
    rng = np.random.default_rng(3)
    src_tok = {0: _tok(sk), 1: _tok(sv)}
    cases = [(l, kv, h, np.sort(rng.choice(w.T, 48, replace=False))) for (l, kv, h) in
             [(0, 0, 0), (0, 1, 7), (21, 0, 3), (40, 1, 5), (63, 0, 7), (63, 1, 2)]]
    _check(w, 1024, sel, P, src_tok, pos.reshape(-1), (tk, tv), cases)


def test_mlp_empty_call_writes_nothing():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4_xhead", Ls=2, Lt=2, H=2, B=1, T=64, k=1)
    dev = torch.device("cuda:0")
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    P = _weights(w, 256, 14, dev)
    tk = torch.full((w.Lt, w.B, w.H, w.T, w.d), 7.0, dtype=torch.bfloat16, device=dev)
    tv = tk.clone()
    pos = torch.from_numpy(syn.positions(w)).to(dev)
    cfg = kvx.mlp_config(w.Ls, w.Lt, w.H, w.d, w.k, 256, w.theta_s, w.theta_t, sel,
                         *(P[n].data_ptr() for n in ("W1", "b1", "W2", "b2", "W3", "b3")))
    for (B, T) in [(0, w.T), (w.B, 0)]:
        kvx.kvx_mlp_map(cfg, kvx.src_from_tensors(sk, sv), B, T, pos.data_ptr(), kvx.tgt_from_tensors(tk, tv),
                        torch.cuda.current_stream().cuda_stream)
    assert torch.all(tk == 7.0) and torch.all(tv == 7.0)


def test_mlp_hf_rope_numerics():
    """KVX_ROPE_HF on the MLP mapper (the Hugging Face forward's rounding in the key strip and
    the target rotation): against the oracle in the same numerics at positions past
    2 * 10^4, 99 % of outputs within 2^-7 of the block RMS, and the keys closer to it on
    average than to the exact-RoPE oracle."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4_xhead", Ls=3, Lt=2, H=2, B=1, T=256, k=2, theta_t=5e5)
    dev = torch.device("cuda:0")
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    pos = syn.positions(w) + 20011
    P = _weights(w, 256, 15, dev)
    tk = torch.full((w.Lt, w.B, w.H, w.T, w.d), float("nan"), dtype=torch.bfloat16, device=dev)
    tv = torch.full_like(tk, float("nan"))
    posd = torch.from_numpy(pos).to(dev)
    cfg = kvx.mlp_config(w.Ls, w.Lt, w.H, w.d, w.k, 256, w.theta_s, w.theta_t, sel,
                         *(P[n].data_ptr() for n in ("W1", "b1", "W2", "b2", "W3", "b3")),
                         rope_numerics=kvx.KVX_ROPE_HF)
    kvx.kvx_mlp_map(cfg, kvx.src_from_tensors(sk, sv), w.B, w.T, posd.data_ptr(), kvx.tgt_from_tensors(tk, tv),
                    torch.cuda.current_stream().cuda_stream)
    params = {n: _dec(P[n]) if P[n].dtype == torch.bfloat16 else P[n].cpu().double().numpy() for n in P}
    args = (_tok(sk), _tok(sv), pos.reshape(-1), sel, params, w.theta_s, w.theta_t, "bf16fwd")
    hk, hv = omlp.map_tokens_mlp(*args, rope_numerics="hf")
    ek, _ = omlp.map_tokens_mlp(*args)
    gk = _dec(tk).transpose(0, 2, 1, 3, 4).reshape(w.Lt, w.H, w.B * w.T, w.d)
    gv = _dec(tv).transpose(0, 2, 1, 3, 4).reshape(w.Lt, w.H, w.B * w.T, w.d)
    for g, r in ((gk, hk), (gv, hv)):
        rms = np.sqrt(np.mean(r * r))
        assert np.mean(np.abs(g - r) <= 2.0 ** -7 * rms) >= 0.99
    assert np.mean(np.abs(gk - hk)) < 0.8 * np.mean(np.abs(gk - ek)), (np.mean(np.abs(gk - hk)), np.mean(np.abs(gk - ek)))
