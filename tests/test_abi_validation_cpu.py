"""Argument validation of the C ABI's host-side entry points, at every boundary (CPU).

Each bound is checked from both sides: the first rejected value and the first accepted
one, one argument at a time with the others valid.  A kvx_create config that passes the
host checks goes on to the device: without a GPU that is KVX_ERR_CUDA (the first CUDA
call fails), with one it is a context, destroyed at once."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_03893_gb300 import build as kbuild
from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn


@pytest.fixture(scope="module", autouse=True)
def built():
    kbuild.build()
    kvx.lib()


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


# ----------------------------------------------------------------- mapper size -------

def test_mapper_params_rejects_each_non_positive_size():
    L = kvx.lib()
    good = [64, 8, 128, 4]
    assert L.kvx_mapper_params(*good, kvx.KVX_PER_HEAD) == 2 * 64 * 8 * 4 * 128 * 128
    for i in range(4):
        for bad in (0, -1):
            args = list(good)
            args[i] = bad
            assert L.kvx_mapper_params(*args, kvx.KVX_PER_HEAD) == -1, (i, bad)
    assert L.kvx_mapper_params(*good, 7) == -1


# ----------------------------------------------------------------- top-k -------------

def test_select_topk_bounds():
    L = kvx.lib()
    S = np.random.default_rng(1).uniform(size=(3, 5))
    out = np.zeros(3 * 5, dtype=np.int32)
    inv = kvx.KVX_ERR_INVALID_ARG
    assert L.kvx_select_topk(None, 3, 5, 2, _ptr(out)) == inv
    assert L.kvx_select_topk(_ptr(S), 3, 5, 2, None) == inv
    assert L.kvx_select_topk(_ptr(S), 0, 5, 2, _ptr(out)) == inv
    assert L.kvx_select_topk(_ptr(S), 3, 0, 2, _ptr(out)) == inv
    assert L.kvx_select_topk(_ptr(S), 3, 5, 0, _ptr(out)) == inv
    assert L.kvx_select_topk(_ptr(S), 3, 5, 6, _ptr(out)) == inv
    assert L.kvx_select_topk(_ptr(S), 3, 5, 1, _ptr(out)) == kvx.KVX_OK
    assert L.kvx_select_topk(_ptr(S), 3, 5, 5, _ptr(out)) == kvx.KVX_OK
    assert np.array_equal(out.reshape(3, 5), np.tile(np.arange(5), (3, 1)))
    for i in range(S.size):                          # a NaN anywhere is refused
        T = S.copy()
        T.flat[i] = np.nan
        assert L.kvx_select_topk(_ptr(T), 3, 5, 2, _ptr(out)) == inv, i


# ----------------------------------------------------------------- kvx_create --------

def _cfg(head_mix="per_head", **over):
    w = syn.workload("tiny_fp32", head_mix=head_mix)
    W, b = syn.weights(w)
    args = dict(src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k,
                theta_s=w.theta_s, theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b,
                scores=syn.selection_scores(w))
    args.update(over)
    cfg, keep = kvx.config_from_tensors(**args)
    if head_mix == "cross_head":
        cfg.head_mix = kvx.KVX_CROSS_HEAD
    return cfg, keep, w


def _create_status(cfg):
    L = kvx.lib()
    out = ctypes.c_void_p()
    st = L.kvx_create(ctypes.byref(cfg), 0, ctypes.byref(out))
    if out.value:
        L.kvx_destroy(out)
    return st, bool(out.value)


def _passes_host_checks(cfg):
    st, made = _create_status(cfg)
    if torch.cuda.is_available():
        return st == kvx.KVX_OK and made
    return st == kvx.KVX_ERR_CUDA and not made


def test_create_accepts_every_valid_enum_and_the_bounds():
    cfg, keep, w = _cfg()
    assert _passes_host_checks(cfg)
    for k in (1, w.Ls):                              # both ends of [1, L_s]
        cfg, keep, w = _cfg(k=k)
        assert _passes_host_checks(cfg), k
    cfg, keep, w = _cfg(head_mix="cross_head")
    assert _passes_host_checks(cfg)
    for field, values in (("rope_style", (kvx.KVX_ROPE_HALF, kvx.KVX_ROPE_INTERLEAVED)),
                          ("rope_numerics", (kvx.KVX_ROPE_EXACT, kvx.KVX_ROPE_HF))):
        for v in values:
            cfg, keep, w = _cfg()
            setattr(cfg, field, v)
            assert _passes_host_checks(cfg), (field, v)
    # theta just above 1 on either side
    for field in ("src_rope_theta", "tgt_rope_theta"):
        cfg, keep, w = _cfg()
        setattr(cfg, field, 1.0 + 1e-9)
        assert _passes_host_checks(cfg), field


def test_create_accepts_head_dim_256_and_bf16_weights():
    w = syn.workload("tiny_fp32", d=256)
    W, b = syn.weights(w)
    cfg, keep = kvx.config_from_tensors(src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=256, k=w.k,
                                        theta_s=w.theta_s, theta_t=w.theta_t, cache_dtype=w.cache_dtype,
                                        W=W, b=b, scores=syn.selection_scores(w))
    assert _passes_host_checks(cfg)
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=3, Lt=2, H=2, B=1, T=16, k=2)
    W, b = syn.weights(w)
    cfg, keep = kvx.config_from_tensors(src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k,
                                        theta_s=w.theta_s, theta_t=w.theta_t, cache_dtype=w.cache_dtype,
                                        W=W, b=b, scores=syn.selection_scores(w))
    assert cfg.weight_dtype == kvx.KVX_BF16 and _passes_host_checks(cfg)


@pytest.mark.parametrize("field", ["src_layers", "tgt_layers", "n_kv_heads", "head_dim"])
def test_create_rejects_each_zero_size(field):
    cfg, keep, w = _cfg()
    setattr(cfg, field, 0)
    st, made = _create_status(cfg)
    assert st == kvx.KVX_ERR_INVALID_ARG and not made


def test_create_rejects_theta_one_and_missing_selection():
    for field in ("src_rope_theta", "tgt_rope_theta"):
        cfg, keep, w = _cfg()
        setattr(cfg, field, 1.0)
        assert _create_status(cfg) == (kvx.KVX_ERR_INVALID_ARG, False), field
    cfg, keep, w = _cfg()
    cfg.selection_scores = None
    cfg.selection = None
    assert _create_status(cfg) == (kvx.KVX_ERR_INVALID_ARG, False)
    for field in ("cache_dtype", "weight_dtype"):
        cfg, keep, w = _cfg()
        setattr(cfg, field, 2)
        assert _create_status(cfg) == (kvx.KVX_ERR_INVALID_ARG, False), field
    cfg, keep, w = _cfg()
    cfg.rope_numerics = 2
    assert _create_status(cfg)[0] == kvx.KVX_ERR_INVALID_ARG


def test_create_rejects_k_zero_with_an_explicit_selection_and_nan_scores():
    w = syn.workload("tiny_fp32")
    cfg, keep, _ = _cfg(selection=np.array([[0, 1]] * w.Lt, dtype=np.int32), scores=None)
    cfg.k = 0
    assert _create_status(cfg) == (kvx.KVX_ERR_INVALID_ARG, False)
    S = syn.selection_scores(w).copy()
    S[w.Lt - 1, w.Ls - 1] = np.nan                  # the selection itself must fail
    cfg, keep, _ = _cfg(scores=S)
    assert _create_status(cfg) == (kvx.KVX_ERR_INVALID_ARG, False)


def test_create_accepts_an_explicit_selection_with_the_end_layers():
    # rows holding layer 0 and layer L_s - 1, scores absent: the caller's table is used
    w = syn.workload("tiny_fp32")
    sel = np.array([[0, w.Ls - 1]] * w.Lt, dtype=np.int32)
    cfg, keep, _ = _cfg(selection=sel, scores=None)
    assert _passes_host_checks(cfg)
    bad = sel.copy()
    bad[w.Lt - 1] = [w.Ls - 1, w.Ls - 1]             # a repeat in the last row only
    cfg, keep, _ = _cfg(selection=bad, scores=None)
    assert _create_status(cfg) == (kvx.KVX_ERR_INVALID_ARG, False)


# ----------------------------------------------------------------- schedule ----------

def test_load_schedule_bounds():
    L = kvx.lib()
    sel = np.array([[0, 1], [1, 2]], dtype=np.int32)
    n = ctypes.c_int32(0)
    bufs = [np.zeros(4, dtype=np.int32) for _ in range(3)]
    ok = [_ptr(sel), ctypes.byref(n)] + [_ptr(x) for x in bufs]
    inv = kvx.KVX_ERR_INVALID_ARG
    assert L.kvx_tc_load_schedule(ok[0], 3, 2, 2, *ok[1:]) == kvx.KVX_OK
    for i in range(5):                               # each pointer NULL on its own
        args = list(ok)
        args[i] = None
        assert L.kvx_tc_load_schedule(args[0], 3, 2, 2, *args[1:]) == inv, i
    for Ls, Lt, k in ((0, 2, 2), (3, 0, 2), (3, 2, 0), (1, 2, 2)):
        assert L.kvx_tc_load_schedule(ok[0], Ls, Lt, k, *ok[1:]) == inv, (Ls, Lt, k)
    # a repeat is found wherever it sits in the row
    for row in ([1, 2, 1], [2, 1, 1], [1, 1, 2]):
        sel3 = np.array([row], dtype=np.int32)
        assert L.kvx_tc_load_schedule(_ptr(sel3), 3, 1, 3, *ok[1:]) == inv, row


def test_load_schedule_writes_nothing_past_its_tables():
    # every use a new layer: n_loads = L_t k fills the tables exactly
    L = kvx.lib()
    Lt, k = 3, 2
    sel = np.arange(Lt * k, dtype=np.int32).reshape(Lt, k)
    n = ctypes.c_int32(0)
    bufs = [np.full(Lt * k + 4, -7, dtype=np.int32) for _ in range(3)]
    assert L.kvx_tc_load_schedule(_ptr(sel), Lt * k, Lt, k, ctypes.byref(n), *[_ptr(x) for x in bufs]) == kvx.KVX_OK
    assert n.value == Lt * k
    for x in bufs:
        assert np.all(x[Lt * k:] == -7)
