"""Pins for oracle.selection, oracle.r2, oracle.ridge and the mapper-size formula (CPU).

Selection is pinned by brute force over all k-subsets, hand-worked ties and a
chi-square test of uniformity; R^2 by exact linear data (R^2 = 1), the textbook
squared Pearson correlation for one regressor, and an analytic noise level; ridge by
exact recovery of a known linear map as lambda -> 0, the normal equations, the
augmented least-squares formulation solved by numpy's lstsq, scikit-learn's Ridge
where available, and the lambda -> infinity limit; the size formula by the paper's
printed table (tests/golden/mapper_sizes.txt).
"""
import itertools
import os

import numpy as np
import pytest

from oracle import mapper, r2, ridge, selection

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------- selection ---------

def test_topk_equals_brute_force_max_sum_subset():
    rng = np.random.default_rng(11)
    for trial in range(50):
        ls, lt, k = 7, 5, int(rng.integers(1, 5))
        S = rng.uniform(size=(lt, ls))
        sel = selection.select_topk(S, k)
        for l in range(lt):
            best = max(itertools.combinations(range(ls), k), key=lambda c: sum(S[l, list(c)]))
            assert tuple(sel[l]) == tuple(sorted(best))


def test_topk_ties_prefer_lower_index_and_rows_ascend():
    S = np.array([[1.0, 3.0, 3.0, 2.0, 3.0],
                  [5.0, 5.0, 5.0, 5.0, 5.0],
                  [0.0, 9.0, 1.0, 9.0, 1.0]])
    sel = selection.select_topk(S, 2)
    assert sel.tolist() == [[1, 2], [0, 1], [1, 3]]
    sel3 = selection.select_topk(S, 3)
    assert sel3.tolist() == [[1, 2, 4], [0, 1, 2], [1, 2, 3]]


def test_topk_uniform_scores_give_uniform_subsets():
    # L_s = 4, k = 2: six subsets, each with probability 1/6 under iid scores
    counts = {}
    rng = np.random.default_rng(12)
    n = 6000
    sel = selection.select_topk(rng.uniform(size=(n, 4)), 2)
    for row in sel:
        counts[tuple(row)] = counts.get(tuple(row), 0) + 1
    assert len(counts) == 6
    chi2 = sum((c - n / 6) ** 2 / (n / 6) for c in counts.values())
    assert chi2 < 20.5  # 5 dof, p ~ 0.001


def test_topk_of_every_layer_is_every_layer():
    S = np.random.default_rng(3).uniform(size=(5, 4))
    assert np.array_equal(selection.select_topk(S, 4), np.tile(np.arange(4), (5, 1)))


def test_topk_rejects_bad_k():
    with pytest.raises(ValueError):
        selection.select_topk(np.zeros((2, 3)), 4)
    with pytest.raises(ValueError):
        selection.select_topk(np.zeros((2, 3)), 0)


# ----------------------------------------------------------------- R^2 -----------

def test_r2_exact_linear_relation_is_one():
    rng = np.random.default_rng(13)
    X = rng.standard_normal((500, 6))
    Y = X @ rng.standard_normal((6, 4)) + rng.standard_normal(4)
    assert abs(r2.r2_ols(X, Y) - 1.0) < 1e-12


def test_r2_single_regressor_is_squared_pearson():
    rng = np.random.default_rng(14)
    x = rng.standard_normal(400)
    y = 0.7 * x + rng.standard_normal(400)
    rho = np.corrcoef(x, y)[0, 1]
    assert abs(r2.r2_ols(x[:, None], y[:, None]) - rho ** 2) < 1e-12


def test_r2_noise_level_and_pooling():
    # channel 0 fully explained, channel 1 pure noise of the same variance: pooled 0.5
    rng = np.random.default_rng(15)
    N = 200000
    X = rng.standard_normal((N, 3))
    Y = np.stack([X @ np.array([1.0, 0.0, 0.0]), rng.standard_normal(N)], axis=1)
    assert abs(r2.r2_ols(X, Y) - 0.5) < 0.01


def test_head_averaged_r2_and_scores():
    rng = np.random.default_rng(16)
    N, d = 300, 4
    src = rng.standard_normal((2, N, d))              # 2 heads
    tgt = np.stack([src[0] @ rng.standard_normal((d, d)), rng.standard_normal((N, d))])
    h = r2.head_averaged_r2(src, tgt)
    assert abs(h - 0.5 * (1.0 + r2.r2_ols(src[1], tgt[1]))) < 1e-12
    S = r2.selection_scores([src, src], [src, src], [tgt], [tgt])
    assert S.shape == (1, 2) and abs(S[0, 0] - h) < 1e-12



def test_r2_matrix_and_scores_find_planted_sources():
    # L_s = 3 source layers, L_t = 2 target layers, H = 2 heads (sizes differ, so a
    # transposed index fails).  Keys of target layer l are an exact linear map of source
    # layer sigma(l), values of source layer tau(l) != sigma(l); every other layer is
    # independent.  Per-head regression: target head 1 of layer 1 depends only on source
    # head 0, which a same-head probe must not see.
    rng = np.random.default_rng(21)
    N, d, Ls, Lt, H = 2000, 3, 3, 2, 2
    srcK = rng.standard_normal((Ls, H, N, d))
    srcV = rng.standard_normal((Ls, H, N, d))
    sigma, tau = [2, 0], [1, 2]
    tgtK = np.stack([np.stack([srcK[sigma[l], h] @ rng.standard_normal((d, d)) + 0.3 for h in range(H)])
                     for l in range(Lt)])
    # values map d = 3 source channels to 2 target channels: the target is explained
    # exactly, while a regression the other way round (source on target) could not be
    tgtV = np.stack([np.stack([srcV[tau[l], h] @ rng.standard_normal((d, d - 1)) for h in range(H)])
                     for l in range(Lt)])
    tgtK[1, 1] = srcK[sigma[1], 0] @ rng.standard_normal((d, d))     # the other source head
    RK, RV = r2.r2_matrix(srcK, tgtK), r2.r2_matrix(srcV, tgtV)
    assert RK.shape == (Lt, Ls) and RV.shape == (Lt, Ls)
    noise = 5.0 * d / N                                   # R^2 of unrelated data is ~ d / N
    for l in range(Lt):
        for lp in range(Ls):
            assert (abs(RV[l, lp] - 1.0) < 1e-10) if lp == tau[l] else (RV[l, lp] < noise)
    assert abs(RK[0, sigma[0]] - 1.0) < 1e-10
    # layer 1: head 0 is exact, head 1 only through the other head: R^2 ~ 1/2
    assert abs(RK[1, sigma[1]] - 0.5) < noise
    assert all(RK[l, lp] < noise for l in range(Lt) for lp in range(Ls) if lp != sigma[l])
    S = r2.selection_scores(srcK, srcV, tgtK, tgtV)
    assert np.allclose(S, 0.5 * (RK + RV), rtol=0, atol=1e-15)
    # the planted layers are the top two of each target layer, in the paper's order
    assert [sorted(np.argsort(-S[l])[:2].tolist()) for l in range(Lt)] == \
        [sorted([sigma[l], tau[l]]) for l in range(Lt)]


# ----------------------------------------------------------------- ridge ---------

def _linear_data(seed, N=400, F=12, d=5, noise=0.0):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((N, F)) * rng.uniform(0.5, 2.0, F) + rng.standard_normal(F)
    W0 = rng.standard_normal((F, d))
    b0 = rng.standard_normal(d)
    Y = X @ W0 + b0 + noise * rng.standard_normal((N, d))
    return X, Y, W0, b0


def test_ridge_recovers_known_map_as_lambda_vanishes():
    X, Y, W0, b0 = _linear_data(17)
    W, b = ridge.fit_ridge(X, Y, lam=1e-10)
    assert np.max(np.abs(W - W0)) < 1e-8
    assert np.max(np.abs(b - b0)) < 1e-8


def test_ridge_normal_equations_and_bias_identity():
    X, Y, _, _ = _linear_data(18, noise=0.3)
    lam = 0.01
    W, b = ridge.fit_ridge(X, Y, lam)
    Xc, Yc = X - X.mean(0), Y - Y.mean(0)
    resid = (Xc.T @ Xc + lam * np.eye(X.shape[1])) @ W - Xc.T @ Yc
    assert np.max(np.abs(resid)) < 1e-9
    assert np.max(np.abs(b - (Y.mean(0) - X.mean(0) @ W))) < 1e-12


def test_ridge_equals_augmented_least_squares():
    X, Y, _, _ = _linear_data(19, N=60, F=20, noise=1.0)
    lam = 3.0
    W, _ = ridge.fit_ridge(X, Y, lam)
    Xc, Yc = X - X.mean(0), Y - Y.mean(0)
    A = np.vstack([Xc, np.sqrt(lam) * np.eye(X.shape[1])])
    B = np.vstack([Yc, np.zeros((X.shape[1], Y.shape[1]))])
    W_ls, *_ = np.linalg.lstsq(A, B, rcond=None)
    assert np.max(np.abs(W - W_ls)) < 1e-10


def test_ridge_matches_sklearn():
    linear_model = pytest.importorskip("sklearn.linear_model")
    X, Y, _, _ = _linear_data(20, N=80, F=15, noise=0.5)
    W, b = ridge.fit_ridge(X, Y, 0.7)
    m = linear_model.Ridge(alpha=0.7, fit_intercept=True, solver="svd").fit(X, Y)
    assert np.max(np.abs(W - m.coef_.T)) < 1e-9
    assert np.max(np.abs(b - m.intercept_)) < 1e-9


def test_ridge_large_lambda_limit():
    X, Y, _, _ = _linear_data(21, noise=0.5)
    W, b = ridge.fit_ridge(X, Y, lam=1e14)
    assert np.max(np.abs(W)) < 1e-9
    assert np.max(np.abs(b - Y.mean(0))) < 1e-7


# ------------------------------------------------------- mapper-size formula -----

def test_mapper_params_reproduce_papers_table():
    rows = [ln.split() for ln in open(os.path.join(GOLDEN, "mapper_sizes.txt"))
            if ln.strip() and not ln.startswith("#")]
    assert len(rows) == 6
    for name, k, lt, nkv, dh, params_b, storage_gb in rows:
        p = mapper.mapper_params(int(lt), int(nkv), int(dh), int(k), head_mix="cross_head")
        assert round(p / 1e9, 2) == float(params_b), name
        # storage: fp32 parameters, printed in GiB rounded to a whole number
        assert abs(p * 4 / 2 ** 30 - float(storage_gb)) <= 0.5, name


def test_mapper_params_per_head():
    assert mapper.mapper_params(64, 8, 128, 4, head_mix="per_head") == 2 * 64 * 8 * 512 * 128
