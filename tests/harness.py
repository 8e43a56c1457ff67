"""Test-side glue: run the CUDA path through the C ABI and the oracle on the same
seeded inputs, and compare with the stated tolerances.

Tolerances (the mapped output of a workload is compared element by element):
* fp32 caches: max |gpu - ref| <= 1e-4 * RMS(ref), ref in the oracle's "exact" mode;
* bf16 caches: |gpu - ref| <= 2^-7 |ref| + 1e-3 RMS(ref) for every element, ref in the
  oracle's "bf16fwd" mode (stripped keys rounded to bf16 before the contraction).
RMS(ref) is taken over every compared element of K and V together.

bf16 keys also get the oracle's rounding slack: the kernels strip the source RoPE in
fp32 (angle error below 1e-6 rad, sincosf within 2 ulp, two roundings), so a stripped
key x of the pair (a, b) is known to within STRIP_DELTA (|a| + |b|).  Where that
interval straddles a bf16 rounding midpoint either neighbour is a correct bf16-forward
operand, and the bound of that output grows by the oracle's worst-case contribution of
the other choice.  Elements with no such key compare at the plain tolerance.
"""
import numpy as np
import torch

from oracle import bf16 as obf16
from oracle import mapper as omap
from oracle import rope as orope
from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn

BF16_REL = 2.0 ** -7
BF16_ABS_RMS = 1e-3
F32_ABS_RMS = 1e-4
STRIP_DELTA = 4e-6


def to_f64(t):
    """Exact float64 copy of a CPU/GPU tensor of float32 or bfloat16."""
    t = t.detach().contiguous().cpu()
    if t.dtype == torch.bfloat16:
        return obf16.decode(t.view(torch.int16).numpy().view(np.uint16))
    return t.numpy().astype(np.float64)


def rope_theta(w, side):
    """The oracle's RoPE base for one side of a workload (a RopeSpec when it is scaled)."""
    theta = w.theta_s if side == 0 else w.theta_t
    if not w.rope_scaling:
        return theta
    return orope.RopeSpec(theta, orope.Llama3Scaling(*w.rope_scaling))


def make_ctx(w, kernel=kvx.KVX_KERNEL_AUTO, selection=None, W=None, b=None, scores=None,
             device=0, rope_style=None):
    if rope_style is None:   # the workload's pairing unless the test asks for another
        rope_style = kvx.KVX_ROPE_INTERLEAVED if w.rope_style == "interleaved" else kvx.KVX_ROPE_HALF
    if W is None:
        W, b = syn.weights(w)
    if selection is None and scores is None:
        scores = syn.selection_scores(w)
    cfg, keep = kvx.config_from_tensors(
        src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k,
        theta_s=w.theta_s, theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b,
        selection=selection, scores=scores, rope_style=rope_style,
        head_mix=kvx.KVX_CROSS_HEAD if w.head_mix == "cross_head" else kvx.KVX_PER_HEAD,
        rope_scaling=w.rope_scaling or None)
    ctx = kvx.kvx_create(cfg, device)
    if kernel != kvx.KVX_KERNEL_AUTO:
        kvx.kvx_set_kernel(ctx, kernel)
    sel = kvx.kvx_get_selection(ctx, w.Lt, w.k)
    return ctx, sel, W, b


def run_contiguous(ctx, w, sk, sv, pos_np, out_dtype=None, tgt=None):
    dev = sk.device
    pos = torch.from_numpy(np.ascontiguousarray(pos_np, dtype=np.int32)).to(dev)
    B, T = pos_np.shape
    if tgt is None:
        dt = out_dtype or sk.dtype
        tk = torch.full((w.Lt, B, w.H, T, w.d), float("nan"), dtype=dt, device=dev)
        tv = torch.full_like(tk, float("nan"))
    else:
        tk, tv = tgt
    stream = torch.cuda.current_stream().cuda_stream
    kvx.kvx_map(ctx, kvx.src_from_tensors(sk, sv), B, T, pos.data_ptr(),
                kvx.tgt_from_tensors(tk, tv), stream)
    status = kvx.kvx_get_status(ctx, stream)
    return tk, tv, status


def oracle_full(w, sk, sv, pos_np, sel, W, b, style=None):
    """Returns (ref_k, ref_v, slack_k, slack_v); style None = the workload's RoPE pairing."""
    style = style or w.rope_style
    mode = "exact" if w.cache_dtype == "f32" else "bf16fwd"
    return omap.map_cache(to_f64(sk), to_f64(sv), pos_np, sel, to_f64(W),
                          None if b is None else to_f64(b), rope_theta(w, 0), rope_theta(w, 1), mode=mode,
                          style=style, head_mix=w.head_mix, rounding_slack=STRIP_DELTA)


def check(w, got, ref, slack=None):
    """got/ref/slack: lists of float64 arrays of equal shapes.
    Returns (ok, worst err/bound, rms, number of failing elements)."""
    g = np.concatenate([x.ravel() for x in got])
    r = np.concatenate([x.ravel() for x in ref])
    rms = float(np.sqrt(np.mean(r * r)))
    err = np.abs(g - r)
    if w.cache_dtype == "f32":
        bound = F32_ABS_RMS * rms + 0 * r
    else:
        bound = BF16_REL * np.abs(r) + BF16_ABS_RMS * rms
        if slack is not None:
            bound = bound + np.concatenate([x.ravel() for x in slack])
    bad = ~(err <= bound)          # NaN counts as a failure
    ratio = float(np.max(err / bound)) if np.all(np.isfinite(err)) else float("inf")
    return (not bad.any()), ratio, rms, int(bad.sum())


def sample_rows(w, n, seed=0, turn_T=None):
    """Token rows (b, t) to check at full size: first and last tiles, tile borders,
    the ragged tail and random rows."""
    T = w.T if turn_T is None else turn_T
    rng = np.random.default_rng(1000 + seed)
    fixed = [(0, 0), (0, 1), (0, 127), (0, 128), (w.B - 1, T - 1), (w.B - 1, T - 2),
             (w.B - 1, (T - 1) // 128 * 128)]
    rand = [(int(rng.integers(0, w.B)), int(rng.integers(0, T))) for _ in range(n)]
    rows = sorted(set((b, t) for b, t in fixed + rand if 0 <= t < T))
    return np.array(rows, dtype=np.int64)


def oracle_rows(w, rows, pos_np, sel, W, b, turn=None):
    """Oracle output at chosen token rows: returns (ref_k, ref_v, slack_k, slack_v),
    each [L_t][H][n][d]."""
    mode = "exact" if w.cache_dtype == "f32" else "bf16fwd"
    sk = to_f64(syn.source_rows(w, 0, rows, turn=turn))
    sv = to_f64(syn.source_rows(w, 1, rows, turn=turn))
    p = pos_np[rows[:, 0], rows[:, 1]]
    return omap.map_tokens(sk, sv, p, sel, to_f64(W), None if b is None else to_f64(b),
                           rope_theta(w, 0), rope_theta(w, 1), mode=mode, head_mix=w.head_mix,
                           style=w.rope_style, rounding_slack=STRIP_DELTA)
