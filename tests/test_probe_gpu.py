"""GPU parity of the single-source R^2 probe (kvx_r2_probe, Sec. 2.3 and Sec. 3.2) and of the
device top-k (kvx_select_topk_device) against the float64 oracle (oracle.r2 on
RoPE-stripped features built with oracle.rope), on seeded synthetic caches.

Tolerance (derived from the arithmetic): the centred cross-products A = Xc^T Xc and
C = Xc^T Yc carry a relative error of at most eps = N u + 2^-16 (u = 2^-24; fp32
accumulation of products of bf16 hi + lo operands within 2^-17 of the values) of their
Cauchy-Schwarz scale.  R^2 = tr(C^T A^{-1} C) / SS_tot is then perturbed by at most about
(kappa + 2) eps, kappa the condition number of the source Gram block scaled to unit
diagonal; the fp32 product L^{-1} C adds about 128 u sqrt(kappa).  The test bound on each
head-averaged R^2 is 8 ((kappa + 2) eps + 128 u sqrt(kappa)), kappa the largest over heads."""
import numpy as np
import pytest
import torch

from oracle import bf16 as obf16
from oracle import r2 as or2
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


def _f64(t):
    return obf16.decode(t.cpu().view(torch.int16).numpy().view(np.uint16))


def _layer_features(cache, layer, kv, theta, pos):
    """Layer `layer` of a [L][B][H][T][d] cache -> float64 [H][N][d], keys RoPE-stripped."""
    x = _f64(cache[layer])
    B, H, T, d = x.shape
    x = x.transpose(1, 0, 2, 3).reshape(H, B * T, d)
    if kv == 0:
        x = orope.rotate(x, pos.reshape(-1)[None, :], theta, inverse=True)
    return x


def _mixed_targets(w, sk, sv, gen):
    """Target layer l = 0.8 src[a_l] + 0.5 src[b_l] + 0.4 noise (same heads, same positions),
    rounded to bf16: with theta_t = theta_s the stripped target keys are the same mixture of
    the stripped source keys, so the probe has clear winners."""
    out = []
    picks = []
    for kvc in (sk, sv):
        layers = []
        for l in range(w.Lt):
            a, b = l % w.Ls, (l + 2) % w.Ls
            if kvc is sk:
                picks.append((a, b))
            noise = torch.randn(kvc.shape[1:], generator=gen, device="cpu").to(kvc.device)
            y = 0.8 * kvc[a].float() + 0.5 * kvc[b].float() + 0.4 * noise
            layers.append(y.to(torch.bfloat16))
        out.append(torch.stack(layers).contiguous())
    return out[0], out[1], picks


def _run_probe(w, sk, sv, tk, tv, pos):
    dev = sk.device
    posd = torch.from_numpy(pos).to(dev)
    scores = torch.full((w.Lt, w.Ls), float("nan"), dtype=torch.float64, device=dev)
    r2kv = torch.full((2, w.Lt, w.Ls), float("nan"), dtype=torch.float64, device=dev)
    s = torch.cuda.current_stream().cuda_stream
    kvx.kvx_r2_probe(w.Ls, w.Lt, w.H, w.d, w.theta_s, w.theta_t, kvx.src_from_tensors(sk, sv),
                     kvx.src_from_tensors(tk, tv), w.B, w.T, posd.data_ptr(), scores.data_ptr(), r2kv.data_ptr(), s)
    return scores, r2kv


def _kappa_scaled(X):
    Xc = X - X.mean(axis=0)
    A = Xc.T @ Xc
    dg = np.sqrt(np.diag(A))
    return np.linalg.cond(A / np.outer(dg, dg))


def _tolerance(N, kappa):
    eps = N * U + 2.0 ** -16
    return 8.0 * ((kappa + 2.0) * eps + 128 * U * np.sqrt(kappa))


def _check_pairs(w, sk, sv, tk, tv, pos, r2kv, pairs):
    N = w.B * w.T
    feats = {}

    def feat(side, kv, layer):
        key = (side, kv, layer)
        if key not in feats:
            cache = (sk if kv == 0 else sv) if side == 0 else (tk if kv == 0 else tv)
            feats[key] = _layer_features(cache, layer, kv, w.theta_s if side == 0 else w.theta_t, pos)
        return feats[key]

    kap = {}
    g = r2kv.cpu().numpy()
    worst = 0.0
    for (l, s) in pairs:
        for kv in (0, 1):
            xs, xt = feat(0, kv, s), feat(1, kv, l)
            ref = or2.head_averaged_r2(xs, xt)
            if (kv, s) not in kap:
                kap[(kv, s)] = max(_kappa_scaled(xs[h]) for h in range(w.H))
            tol = _tolerance(N, kap[(kv, s)])
            err = abs(g[kv, l, s] - ref)
            worst = max(worst, err / tol)
            assert err <= tol, "R2 kv=%d (t=%d, s=%d): gpu %.9f ref %.9f err %.3g > %.3g" % (
                kv, l, s, g[kv, l, s], ref, err, tol)
    return worst


@pytest.mark.parametrize("over,mixed", [
    (dict(Ls=5, Lt=4, H=2, B=2, T=300, theta_t=1e6), True),      # structured: clear winners, ragged chunk
    (dict(Ls=4, Lt=3, H=1, B=1, T=700, theta_t=5e5), False),     # independent targets, different thetas
    (dict(Ls=3, Lt=5, H=2, B=3, T=100), False),                  # B > 1, short sequences
])
def test_probe_small_every_pair(over, mixed):
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", **over)
    dev = torch.device("cuda:0")
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    if mixed:
        gen = torch.Generator().manual_seed(1234)
        tk, tv, picks = _mixed_targets(w, sk, sv, gen)
    else:
        tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = syn.positions(w)
    scores, r2kv = _run_probe(w, sk, sv, tk, tv, pos)
    sc = scores.cpu().numpy()
    assert np.all(np.isfinite(sc)), "unwritten scores"
    assert np.allclose(sc, 0.5 * (r2kv[0] + r2kv[1]).cpu().numpy(), rtol=0, atol=1e-15)
    pairs = [(l, s) for l in range(w.Lt) for s in range(w.Ls)]
    _check_pairs(w, sk, sv, tk, tv, pos, r2kv, pairs)
    # device top-k of the GPU scores = host top-k of the same scores (bit-exact)
    k = min(2, w.Ls)
    sel_d = torch.empty((w.Lt, k), dtype=torch.int32, device=dev)
    kvx.kvx_select_topk_device(scores.data_ptr(), w.Lt, w.Ls, k, sel_d.data_ptr(),
                               torch.cuda.current_stream().cuda_stream)
    sel_h = kvx.kvx_select_topk(sc, k)
    assert np.array_equal(sel_d.cpu().numpy(), np.asarray(sel_h).reshape(w.Lt, k))
    if mixed:   # the two mixed-in source layers win every row
        for l, (a, b) in enumerate(picks):
            assert sorted(sel_d[l].tolist()) == sorted([a, b]), (l, a, b, sc[l])


def test_probe_headline_shapes_sampled():
    """Qwen3-14B -> 32B layer and head counts, 2048 calibration tokens: every (target, source)
    pair scored on the GPU, twelve pairs checked against the oracle, the full score matrix
    checked for range and for the identity score = mean of K and V."""
    w = syn.workload("qwen3_14b_32b_t32768_k4", T=2048)
    dev = torch.device("cuda:0")
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = syn.positions(w)
    scores, r2kv = _run_probe(w, sk, sv, tk, tv, pos)
    sc = scores.cpu().numpy()
    assert np.all(np.isfinite(sc)) and np.all(sc >= -1e-6) and np.all(sc <= 1 + 1e-6)
    pairs = [(0, 0), (0, 39), (7, 13), (21, 5), (31, 20), (40, 33), (47, 1), (52, 26), (58, 38), (63, 0),
             (63, 17), (63, 39)]
    _check_pairs(w, sk, sv, tk, tv, pos, r2kv, pairs)


def test_select_topk_device_matches_host_on_tie_heavy_scores():
    rng = np.random.default_rng(7)
    dev = torch.device("cuda:0")
    for (lt, ls, k) in [(64, 40, 4), (80, 32, 3), (5, 7, 7), (1, 1, 1), (300, 126, 8)]:
        sc = rng.integers(0, 4, size=(lt, ls)).astype(np.float64)   # many ties
        d = torch.from_numpy(sc).to(dev)
        out = torch.empty((lt, k), dtype=torch.int32, device=dev)
        kvx.kvx_select_topk_device(d.data_ptr(), lt, ls, k, out.data_ptr(), torch.cuda.current_stream().cuda_stream)
        ref = np.asarray(kvx.kvx_select_topk(sc, k)).reshape(lt, k)
        assert np.array_equal(out.cpu().numpy(), ref), (lt, ls, k)


def test_select_topk_device_reports_nan():
    dev = torch.device("cuda:0")
    sc = torch.zeros((3, 4), dtype=torch.float64, device=dev)
    sc[1, 2] = float("nan")
    out = torch.empty((3, 2), dtype=torch.int32, device=dev)
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_select_topk_device(sc.data_ptr(), 3, 4, 2, out.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_probe_caller_workspace():
    """kvx_r2_probe with a caller workspace of kvx_r2_probe_workspace_bytes: scores
    bit-identical to the call's own allocation; a small workspace (tokens in chunks) stays
    within the oracle tolerance; one below the fixed pieces is refused."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=4, Lt=3, H=2, B=2, T=300)
    dev = torch.device("cuda:0")
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = syn.positions(w)
    scores0, r2kv0 = _run_probe(w, sk, sv, tk, tv, pos)
    args = (w.Ls, w.Lt, w.H, w.d, w.theta_s, w.theta_t)
    full = kvx.kvx_r2_probe_workspace_bytes(*args, w.B, w.T)
    per64 = kvx.kvx_r2_probe_workspace_bytes(*args, 1, 128) - kvx.kvx_r2_probe_workspace_bytes(*args, 1, 64)
    posd = torch.from_numpy(pos).to(dev)
    s = torch.cuda.current_stream().cuda_stream

    def probe(nbytes):
        ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        sc = torch.full((w.Lt, w.Ls), float("nan"), dtype=torch.float64, device=dev)
        r2 = torch.full((2, w.Lt, w.Ls), float("nan"), dtype=torch.float64, device=dev)
        kvx.kvx_r2_probe(*args, kvx.src_from_tensors(sk, sv), kvx.src_from_tensors(tk, tv), w.B, w.T,
                         posd.data_ptr(), sc.data_ptr(), r2.data_ptr(), s, workspace_ptr=ws.data_ptr(),
                         workspace_bytes=nbytes)
        return sc, r2

    sc1, r21 = probe(full)
    assert torch.equal(sc1, scores0) and torch.equal(r21, r2kv0)
    n_chunks_tokens = (w.B * w.T + 63) // 64 * 64
    sc2, r22 = probe(full - (n_chunks_tokens // 64 - 2) * per64)      # two 64-token columns: chunks
    pairs = [(l, s_) for l in range(w.Lt) for s_ in range(w.Ls)]
    _check_pairs(w, sk, sv, tk, tv, pos, r22, pairs)
    with pytest.raises(kvx.KvxError) as e:
        probe(4096)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_probe_reports_a_singular_source_block():
    """A constant channel makes a centred source Gram block singular: the probe reports
    INVALID_ARG instead of returning scores (OLS has no unique fit there)."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=3, Lt=2, H=1, B=1, T=300)
    dev = torch.device("cuda:0")
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    sv[1, :, :, :, 5] = 0.75                      # value channel 5 of source layer 1: constant
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    with pytest.raises(kvx.KvxError) as e:
        _run_probe(w, sk, sv, tk, tv, syn.positions(w))
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    assert "singular" in kvx.lib().kvx_last_error().decode()
