"""Top-k source-layer selection (oracle; test infrastructure only).

Sec. 3.2 (cross-layer source selection): for each target layer l the k source layers
with the highest score S[l][l'] (head-averaged R^2, averaged over RoPE-stripped keys
and values) are selected; every head of layer l shares them.

Readings where the paper is silent: ties go to the lower source index, and the
selected layers are listed in ascending source-layer order, which is also the order of
the row blocks of W (the concatenation order of Sec. 3.2).
"""
import numpy as np


def select_topk(scores, k):
    """scores: float64 [L_t][L_s] -> int32 [L_t][k], each row ascending."""
    s = np.asarray(scores, dtype=np.float64)
    lt, ls = s.shape
    if not 1 <= k <= ls:
        raise ValueError("k out of range")
    out = np.empty((lt, k), dtype=np.int32)
    idx = np.arange(ls)
    for l in range(lt):
        # primary key: score descending; secondary: source index ascending
        order = np.lexsort((idx, -s[l]))
        out[l] = np.sort(order[:k])
    return out
