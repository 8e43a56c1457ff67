"""Centred closed-form ridge fit (oracle; test infrastructure only).

Sec. 3.1 (per-head ridge regression), Eq. Wstar:  W* = (X^T X + lambda I)^{-1} X^T Y,
computed on X and Y centred by their column means; the bias of Eq. ridge_kv is then
b = mean(Y) - mean(X) W*.  The production lambda is 0.01 (Sec. 3.1).

Reading where the paper is silent: lambda multiplies the identity added to the
*unnormalised* sum X^T X, exactly as Eq. Wstar is written (not a per-sample mean).
The SPD system is solved by a Cholesky factorisation (library primitive).
"""
import numpy as np
import scipy.linalg

LAMBDA_PAPER = 0.01


def fit_ridge(X, Y, lam=LAMBDA_PAPER):
    """X: [N][F], Y: [N][d] (float64).  Returns (W [F][d], b [d])."""
    X = np.asarray(X, dtype=np.float64)
    Y = np.asarray(Y, dtype=np.float64)
    x_mean = X.mean(axis=0)
    y_mean = Y.mean(axis=0)
    Xc = X - x_mean
    Yc = Y - y_mean
    A = Xc.T @ Xc + lam * np.eye(X.shape[1])
    rhs = Xc.T @ Yc
    factor = scipy.linalg.cho_factor(A, lower=True)
    W = scipy.linalg.cho_solve(factor, rhs)
    b = y_mean - x_mean @ W
    return W, b
