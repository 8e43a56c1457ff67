"""Single-source OLS probe and selection scores (oracle; test infrastructure only).

Sec. 2.3 (linear structure), Eq. single_source_ols: for source layer l', target layer l
and head h, an ordinary least-squares fit with intercept
    C_t^{l,h} ~= C_s^{l',h} W + b      (row-vector convention)
over N calibration tokens; fit quality is the coefficient of determination R^2,
averaged over the target's KV heads ("head-averaged R^2").

Sec. 3.2: the selection score of (l, l') is the head-averaged R^2 averaged over
RoPE-stripped keys and values.

Reading where the paper is silent: R^2 of a multi-output fit is pooled over output
channels, R^2 = 1 - sum(SS_res) / sum(SS_tot) (variance explained), not a mean of
per-channel R^2.  The least-squares solve is numpy's ``lstsq`` (library primitive).
"""
import numpy as np


def r2_ols(Xs, Yt):
    """Pooled R^2 of the OLS fit with intercept Yt ~ Xs W + b.  Xs [N][ds], Yt [N][dt]."""
    Xs = np.asarray(Xs, dtype=np.float64)
    Yt = np.asarray(Yt, dtype=np.float64)
    Xc = Xs - Xs.mean(axis=0)
    Yc = Yt - Yt.mean(axis=0)
    W, *_ = np.linalg.lstsq(Xc, Yc, rcond=None)
    resid = Yc - Xc @ W
    return 1.0 - float(np.sum(resid * resid)) / float(np.sum(Yc * Yc))


def head_averaged_r2(src, tgt):
    """src: [H][N][ds] (one source layer), tgt: [H][N][dt] (one target layer).

    Head h of the target is regressed on head h of the source; R^2 averaged over h.
    """
    H = tgt.shape[0]
    return float(np.mean([r2_ols(src[h], tgt[h]) for h in range(H)]))


def r2_matrix(src_layers, tgt_layers):
    """src_layers [L_s][H][N][ds], tgt_layers [L_t][H][N][dt] -> R2 [L_t][L_s]."""
    Lt, Ls = len(tgt_layers), len(src_layers)
    R = np.empty((Lt, Ls), dtype=np.float64)
    for l in range(Lt):
        for lp in range(Ls):
            R[l, lp] = head_averaged_r2(src_layers[lp], tgt_layers[l])
    return R


def selection_scores(src_k_stripped, src_v, tgt_k_stripped, tgt_v):
    """Score S[l][l'] = (R2_Kstripped[l][l'] + R2_V[l][l']) / 2  (Sec. 3.2)."""
    return 0.5 * (r2_matrix(src_k_stripped, tgt_k_stripped) + r2_matrix(src_v, tgt_v))
