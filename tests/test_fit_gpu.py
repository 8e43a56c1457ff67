"""GPU parity of the ridge fit (kvx_fit_ridge, through the C ABI) against the float64 oracle
(oracle.ridge.fit_ridge on RoPE-stripped features built with oracle.rope), on seeded
synthetic calibration caches.

Tolerance (derived from the arithmetic): the GPU forms each centred cross-product from a
bf16 hi + lo split of both factors (hi + lo within 2^-17 of the value, so the product
within about 2^-16 of the exact one; the four partial products are exact on the tensor
cores) and accumulates N of them in fp32, so every entry of Xc^T Xc and Xc^T Yc carries a
relative error of at most about N u + 2^-16 (u = 2^-24) of
the Cauchy-Schwarz scale sqrt(G_ii G_jj); the fp64 factorisation and solves add nothing
comparable.  The solution of the perturbed system then differs by at most kappa(A) times
that normwise relative error, so the test bounds max |W_gpu - W_ref| by
8 kappa (N u + 2^-16) max |W_ref| (+ the same relative bound on the bias, scaled by the
largest feature mean)."""
import numpy as np
import pytest
import torch

from oracle import bf16 as obf16
from oracle import ridge as oridge
from oracle import rope as orope
from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn

pytestmark = pytest.mark.gpu


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


def _features(w, cache, kv, theta, pos):
    """[L][B][H][T][d] cache -> float64 [L][H][N][d] with keys RoPE-stripped."""
    x = _f64(cache)                                   # [L][B][H][T][d]
    L, B, H, T, d = x.shape
    x = x.transpose(0, 2, 1, 3, 4).reshape(L, H, B * T, d)
    if kv == 0:
        x = orope.rotate(x, pos.reshape(-1)[None, None, :], theta, inverse=True)
    return x


def _run_fit(w, lam, sel):
    dev = torch.device("cuda:0")
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = syn.positions(w)
    posd = torch.from_numpy(pos).to(dev)
    F = w.k * w.d
    W = torch.full((w.Lt, 2, w.H, F, w.d), float("nan"), dtype=torch.float32, device=dev)
    b = torch.full((w.Lt, 2, w.H, w.d), float("nan"), dtype=torch.float32, device=dev)
    s = torch.cuda.current_stream().cuda_stream
    kvx.kvx_fit_ridge(w.Ls, w.Lt, w.H, w.d, w.k, w.theta_s, w.theta_t, lam, sel,
                      kvx.src_from_tensors(sk, sv), kvx.src_from_tensors(tk, tv), w.B, w.T,
                      posd.data_ptr(), W.data_ptr(), b.data_ptr(), s)
    return (sk, sv, tk, tv, pos), W.cpu().double().numpy(), b.cpu().double().numpy()


def _check_systems(w, lam, sel, caches, Wg, bg, systems):
    _check_systems_theta(w, w.theta_s, w.theta_t, lam, sel, caches, Wg, bg, systems)


def _check_systems_theta(w, theta_s, theta_t, lam, sel, caches, Wg, bg, systems):
    """theta_s / theta_t: plain bases or oracle.rope.RopeSpec (scaled frequencies)."""
    sk, sv, tk, tv, pos = caches
    feats = {}
    N = w.B * w.T
    for (l, kv, h) in systems:
        if kv not in feats:
            feats[kv] = (_features(w, sk if kv == 0 else sv, kv, theta_s, pos),
                         _features(w, tk if kv == 0 else tv, kv, theta_t, pos))
        xs, xt = feats[kv]
        X = np.concatenate([xs[s, h] for s in sel[l]], axis=-1)
        Y = xt[l, h]
        Wr, br = oridge.fit_ridge(X, Y, lam)
        Xc = X - X.mean(axis=0)
        A = Xc.T @ Xc + lam * np.eye(X.shape[1])
        kappa = np.linalg.cond(A)
        rel = 8.0 * kappa * (N * 2.0 ** -24 + 2.0 ** -16)
        errW = np.max(np.abs(Wg[l, kv, h] - Wr))
        assert errW <= rel * np.max(np.abs(Wr)), \
            "W (%d,%d,%d): err %.3g > %.3g (kappa %.3g)" % (l, kv, h, errW, rel * np.max(np.abs(Wr)), kappa)
        bscale = np.max(np.abs(br)) + np.max(np.abs(X.mean(axis=0))) * np.sum(np.abs(Wr), axis=0).max()
        errb = np.max(np.abs(bg[l, kv, h] - br))
        assert errb <= rel * bscale, "b (%d,%d,%d): err %.3g > %.3g" % (l, kv, h, errb, rel * bscale)


@pytest.mark.parametrize("over,lam", [
    (dict(Ls=4, Lt=3, H=2, B=2, T=300, k=2), 0.01),                 # B > 1, ragged tiles
    (dict(Ls=5, Lt=2, H=2, B=1, T=700, k=3, theta_t=5e5), 1.0),     # different thetas, larger lambda
    (dict(Ls=6, Lt=3, H=1, B=1, T=200, k=4), 0.01),                 # F = 512 > N: lambda keeps it SPD
    (dict(Ls=3, Lt=2, H=2, B=1, T=64, k=1), 0.0),                   # no regularisation, N < F
])
def test_fit_small_every_system(over, lam):
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", **over)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    if lam == 0.0 and w.B * w.T <= w.k * w.d:
        over = dict(over, T=4 * w.k * w.d)                            # keep it positive definite
        w = syn.workload("qwen3_14b_32b_b8x1024_k4", **over)
    caches, Wg, bg = _run_fit(w, lam, sel)
    assert np.all(np.isfinite(Wg)) and np.all(np.isfinite(bg)), "unwritten outputs"
    systems = [(l, kv, h) for l in range(w.Lt) for kv in range(2) for h in range(w.H)]
    _check_systems(w, lam, sel, caches, Wg, bg, systems)


def test_fit_headline_shapes_sampled():
    """Qwen3-14B -> 32B layer and head counts, k = 4, 4096 calibration tokens: every system
    fitted on the GPU, six of them checked against the oracle."""
    w = syn.workload("qwen3_14b_32b_t32768_k4", T=4096)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    caches, Wg, bg = _run_fit(w, 0.01, sel)
    assert np.all(np.isfinite(Wg)) and np.all(np.isfinite(bg))
    systems = [(0, 0, 0), (0, 1, 7), (31, 0, 3), (40, 1, 5), (63, 0, 7), (63, 1, 0)]
    _check_systems(w, 0.01, sel, caches, Wg, bg, systems)


def test_fit_caller_workspace_one_pass_and_chunked():
    """A caller workspace of kvx_fit_workspace_bytes gives the same W and b as the call's own
    allocation (bit-identical: the same single pass); a workspace that holds 128 tokens of
    the packed operands runs the tokens in chunks (fp32 partial blocks added), within the
    oracle tolerance; a workspace below the fixed pieces is refused."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=4, Lt=3, H=2, B=2, T=300, k=2)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    caches, W0, b0 = _run_fit(w, 0.01, sel)
    sk, sv, tk, tv, pos = caches
    dev = torch.device("cuda:0")
    posd = torch.from_numpy(pos).to(dev)
    args = (w.Ls, w.Lt, w.H, w.d, w.k, w.theta_s, w.theta_t, 0.01, sel)
    full = kvx.kvx_fit_workspace_bytes(*args, w.B, w.T)
    per64 = kvx.kvx_fit_workspace_bytes(*args, 1, 128) - kvx.kvx_fit_workspace_bytes(*args, 1, 64)
    assert full > 0 and per64 > 0
    s = torch.cuda.current_stream().cuda_stream
    src, tgt = kvx.src_from_tensors(sk, sv), kvx.src_from_tensors(tk, tv)

    def fit(nbytes):
        ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        F = w.k * w.d
        W = torch.full((w.Lt, 2, w.H, F, w.d), float("nan"), dtype=torch.float32, device=dev)
        b = torch.full((w.Lt, 2, w.H, w.d), float("nan"), dtype=torch.float32, device=dev)
        kvx.kvx_fit_ridge(*args, src, tgt, w.B, w.T, posd.data_ptr(), W.data_ptr(), b.data_ptr(), s,
                          workspace_ptr=ws.data_ptr(), workspace_bytes=nbytes)
        return W.cpu().double().numpy(), b.cpu().double().numpy()

    W1, b1 = fit(full)
    assert np.array_equal(W1, W0) and np.array_equal(b1, b0)
    np_full = (w.B * w.T + 63) // 64 * 64
    W2, b2 = fit(full - (np_full // 64 - 2) * per64)          # two 64-token columns: chunks
    systems = [(l, kv, h) for l in range(w.Lt) for kv in range(2) for h in range(w.H)]
    _check_systems(w, 0.01, sel, caches, W2, b2, systems)
    assert not np.array_equal(W2, W0)          # the chunked run did take another path
    with pytest.raises(kvx.KvxError) as e:
        fit(4096)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_fit_llama3_rope_scaling():
    """The fit strips both sides' keys with the llama3-scaled frequencies: every system of a
    small Llama-3.1-like case at positions past 10^5 against the oracle given the same
    scaling (the features are built with oracle.rope.RopeSpec)."""
    spec = (8.0, 1.0, 4.0, 8192.0)
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=4, Lt=3, H=2, B=1, T=512, k=2, theta_s=5e5, theta_t=5e5)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    dev = torch.device("cuda:0")
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = syn.positions(w) + 150001
    posd = torch.from_numpy(pos).to(dev)
    F = w.k * w.d
    W = torch.full((w.Lt, 2, w.H, F, w.d), float("nan"), dtype=torch.float32, device=dev)
    b = torch.full((w.Lt, 2, w.H, w.d), float("nan"), dtype=torch.float32, device=dev)
    kvx.kvx_fit_ridge(w.Ls, w.Lt, w.H, w.d, w.k, w.theta_s, w.theta_t, 0.01, sel, kvx.src_from_tensors(sk, sv),
                      kvx.src_from_tensors(tk, tv), w.B, w.T, posd.data_ptr(), W.data_ptr(), b.data_ptr(),
                      torch.cuda.current_stream().cuda_stream, rope_scaling=spec)
    rs = orope.RopeSpec(w.theta_s, orope.Llama3Scaling(*spec))
    rt = orope.RopeSpec(w.theta_t, orope.Llama3Scaling(*spec))
    systems = [(l, kv, h) for l in range(w.Lt) for kv in range(2) for h in range(w.H)]
    _check_systems_theta(w, rs, rt, 0.01, sel, (sk, sv, tk, tv, pos), W.cpu().double().numpy(),
                         b.cpu().double().numpy(), systems)


def test_fit_hf_rope_numerics():
    """KVX_ROPE_HF on the fit: both sides' keys are stripped with the Hugging Face forward's
    rounding (oracle.rope.rotate_hf, inverse) before centring; every system of a small case at
    positions past 2 * 10^4 against the oracle's fit of those features."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=4, Lt=3, H=2, B=1, T=512, k=2, theta_t=5e5)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    dev = torch.device("cuda:0")
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = syn.positions(w) + 20011
    posd = torch.from_numpy(pos).to(dev)
    F = w.k * w.d
    W = torch.full((w.Lt, 2, w.H, F, w.d), float("nan"), dtype=torch.float32, device=dev)
    b = torch.full((w.Lt, 2, w.H, w.d), float("nan"), dtype=torch.float32, device=dev)
    kvx.kvx_fit_ridge(w.Ls, w.Lt, w.H, w.d, w.k, w.theta_s, w.theta_t, 0.01, sel, kvx.src_from_tensors(sk, sv),
                      kvx.src_from_tensors(tk, tv), w.B, w.T, posd.data_ptr(), W.data_ptr(), b.data_ptr(),
                      torch.cuda.current_stream().cuda_stream, rope_numerics=kvx.KVX_ROPE_HF)
    Wg, bg = W.cpu().double().numpy(), b.cpu().double().numpy()
    N = w.B * w.T

    def feats(cache, kv, theta):
        x = _f64(cache)
        L, B, H, T, d = x.shape
        x = x.transpose(0, 2, 1, 3, 4).reshape(L, H, B * T, d)
        if kv == 0:
            x = orope.rotate_hf(x, pos.reshape(-1)[None, None, :], theta, inverse=True)
        return x

    for kv in range(2):
        xs = feats(sk if kv == 0 else sv, kv, w.theta_s)
        xt = feats(tk if kv == 0 else tv, kv, w.theta_t)
        for l in range(w.Lt):
            for h in range(w.H):
                X = np.concatenate([xs[s, h] for s in sel[l]], axis=-1)
                Wr, br = oridge.fit_ridge(X, xt[l, h], 0.01)
                Xc = X - X.mean(axis=0)
                kappa = np.linalg.cond(Xc.T @ Xc + 0.01 * np.eye(F))
                rel = 8.0 * kappa * (N * 2.0 ** -24 + 2.0 ** -16)
                err = np.max(np.abs(Wg[l, kv, h] - Wr))
                assert err <= rel * np.max(np.abs(Wr)), (l, kv, h, err, rel * np.max(np.abs(Wr)))


# ------------------------------------------------------------ cross-head fit -----

def _run_fit_xh(w, lam, sel):
    """kvx_fit_ridge with head_mix = KVX_CROSS_HEAD; W [L_t][2][H][k H d][d], b [L_t][2][H][d]."""
    dev = torch.device("cuda:0")
    sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
    tk, tv = syn.target_cache(w, 0, device=dev), syn.target_cache(w, 1, device=dev)
    pos = syn.positions(w)
    posd = torch.from_numpy(pos).to(dev)
    F = w.k * w.H * w.d
    W = torch.full((w.Lt, 2, w.H, F, w.d), float("nan"), dtype=torch.float32, device=dev)
    b = torch.full((w.Lt, 2, w.H, w.d), float("nan"), dtype=torch.float32, device=dev)
    kvx.kvx_fit_ridge(w.Ls, w.Lt, w.H, w.d, w.k, w.theta_s, w.theta_t, lam, sel,
                      kvx.src_from_tensors(sk, sv), kvx.src_from_tensors(tk, tv), w.B, w.T,
                      posd.data_ptr(), W.data_ptr(), b.data_ptr(), torch.cuda.current_stream().cuda_stream,
                      head_mix=kvx.KVX_CROSS_HEAD)
    return (sk, sv, tk, tv, pos), W.cpu().double().numpy(), b.cpu().double().numpy()


def _check_xh_systems(w, lam, sel, caches, Wg, bg, systems):
    """systems: (l, kv).  The oracle's fit of the paper's cross-head feature (every KV head of
    the k selected layers, oracle.mlp.cross_head_features) against every target head of
    layer l at once; every head's W and b within the kappa-scaled bound of the module
    docstring."""
    from oracle import mlp as omlp
    sk, sv, tk, tv, pos = caches
    N = w.B * w.T
    p = pos.reshape(-1)
    def raw(cache, j):          # layer j of a [L][B][H][T][d] cache as float64 [H][N][d], as stored
        x = _f64(cache[j])
        return x.transpose(1, 0, 2, 3).reshape(w.H, N, w.d)

    for (l, kv) in systems:
        src = {j: raw(sk if kv == 0 else sv, j) for j in set(sel[l].tolist())}
        X = omlp.cross_head_features(src, l, sel, kv, p, w.theta_s)                    # keys stripped
        yt = _features(w, (tk if kv == 0 else tv)[l:l + 1], kv, w.theta_t, pos)[0]     # [H][N][d]
        Y = np.concatenate(list(yt), axis=-1)                                          # [N][H d], head-minor
        Wr, br = oridge.fit_ridge(X, Y, lam)
        Xc = X - X.mean(axis=0)
        ev = np.linalg.eigvalsh(Xc.T @ Xc + lam * np.eye(X.shape[1]))
        kappa = ev[-1] / ev[0]
        rel = 8.0 * kappa * (N * 2.0 ** -24 + 2.0 ** -16)
        for h in range(w.H):
            wr, b_r = Wr[:, h * w.d:(h + 1) * w.d], br[h * w.d:(h + 1) * w.d]
            errW = np.max(np.abs(Wg[l, kv, h] - wr))
            assert errW <= rel * np.max(np.abs(wr)), \
                "W (%d,%d,%d): err %.3g > %.3g (kappa %.3g)" % (l, kv, h, errW, rel * np.max(np.abs(wr)), kappa)
            bscale = np.max(np.abs(b_r)) + np.max(np.abs(X.mean(axis=0))) * np.sum(np.abs(wr), axis=0).max()
            errb = np.max(np.abs(bg[l, kv, h] - b_r))
            assert errb <= rel * bscale, "b (%d,%d,%d): err %.3g > %.3g" % (l, kv, h, errb, rel * bscale)


@pytest.mark.parametrize("over,lam", [
    (dict(Ls=4, Lt=3, H=2, B=2, T=300, k=2), 0.01),                 # B > 1, ragged tiles, F = 512
    (dict(Ls=5, Lt=2, H=3, B=1, T=900, k=2, theta_t=5e5), 1.0),     # odd head count, F = 768, larger lambda
    (dict(Ls=6, Lt=2, H=2, B=1, T=640, k=3), 0.01),                 # F = 768 > N: lambda keeps it SPD
])
def test_fit_cross_head_small_every_system(over, lam):
    w = syn.workload("qwen3_14b_32b_b8x1024_k4_xhead", **over)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    caches, Wg, bg = _run_fit_xh(w, lam, sel)
    assert np.all(np.isfinite(Wg)) and np.all(np.isfinite(bg)), "unwritten outputs"
    _check_xh_systems(w, lam, sel, caches, Wg, bg, [(l, kv) for l in range(w.Lt) for kv in range(2)])


def test_fit_cross_head_more_systems_than_sms():
    """More cross-head systems (target layers x K|V) than SMs (160 on a 152-SM GB300): the
    factorisation runs in two waves of per-CTA scratch slots and the solves of each wave
    fill every SM; every output is written, and systems of both waves (the first and last
    of each) match the oracle on every target head."""
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    w = syn.workload("qwen3_14b_32b_b8x1024_k4_xhead", Ls=6, Lt=n_sm // 2 + 4, H=2, B=1, T=400, k=1)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    caches, Wg, bg = _run_fit_xh(w, 0.01, sel)
    assert np.all(np.isfinite(Wg)) and np.all(np.isfinite(bg)), "unwritten outputs"
    assert 2 * w.Lt > n_sm
    last = 2 * w.Lt - 1
    systems = sorted({(s // 2, s % 2) for s in (0, 1, n_sm - 1, n_sm, n_sm + 1, last)})
    _check_xh_systems(w, 0.01, sel, caches, Wg, bg, systems)


def test_fit_cross_head_one_head_equals_per_head():
    """With one KV head the cross-head feature is the per-head one: both modes of the GPU fit
    solve the same systems (different kernels), so they agree within the fit bound."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=4, Lt=3, H=1, B=1, T=700, k=3)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    caches, Wp, bp = _run_fit(w, 0.01, sel)
    _, Wx, bx = _run_fit_xh(w, 0.01, sel)
    scale = np.max(np.abs(Wp))
    assert np.max(np.abs(Wx - Wp)) <= 1e-3 * scale, np.max(np.abs(Wx - Wp)) / scale
    _check_xh_systems(w, 0.01, sel, caches, Wx, bx, [(0, 0), (2, 1)])


def test_fit_cross_head_qwen_shapes_sampled():
    """Qwen3-14B -> 32B layer and head counts, k = 4 (d_s = k n_kv d = 4096, the paper's source
    feature), 8192 calibration tokens: all 128 (layer, K|V) systems fitted on the GPU, three
    checked against the oracle on every target head."""
    w = syn.workload("qwen3_14b_32b_t32768_k4_xhead", T=8192)
    sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
    caches, Wg, bg = _run_fit_xh(w, 0.01, sel)
    assert np.all(np.isfinite(Wg)) and np.all(np.isfinite(bg))
    _check_xh_systems(w, 0.01, sel, caches, Wg, bg, [(0, 0), (33, 1), (63, 0)])
    torch.cuda.empty_cache()
