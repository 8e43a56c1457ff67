"""C-ABI library, host side only (no GPU): it builds, loads, exports every symbol that
include/kvx.h declares, and its host logic (selection, size formula, argument
validation before any CUDA call) matches the oracle and the paper."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import mapper as omap
from oracle import selection as osel
from paper_2608_03893_gb300 import build as kbuild
from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    kbuild.build()
    kvx.lib()


def _declared_functions():
    text = open(os.path.join(ROOT, "include", "kvx.h")).read()
    return sorted(set(re.findall(r"KVX_API\s+[\w\s\*]+?\b(kvx_\w+)\s*\(", text)))


def test_header_declares_the_binding_names():
    decl = _declared_functions()
    assert decl == sorted(kvx.EXPORTED)


def test_library_exports_every_declared_symbol():
    L = kvx.lib()
    for name in _declared_functions():
        assert hasattr(L, name), name
    # and nothing else of ours leaks out
    out = os.popen("nm -D --defined-only %s" % kvx.LIB_PATH).read()
    ours = sorted(set(re.findall(r" T (kvx_\w+)", out)))
    assert ours == _declared_functions()


def test_status_strings():
    for s in range(7):
        assert kvx.kvx_status_string(s).startswith("KVX_")
    assert "unknown" in kvx.kvx_status_string(99)


def test_select_topk_matches_oracle_on_every_workload():
    for name in syn.WORKLOADS:
        w = syn.workload(name)
        S = syn.selection_scores(w)
        assert np.array_equal(kvx.kvx_select_topk(S, w.k), osel.select_topk(S, w.k)), name
    # the swept k of the headline shape
    w = syn.workload("qwen3_14b_32b_t32768_k4")
    S = syn.selection_scores(w)
    for k in (1, 2, 3, 4, 7, 40):
        assert np.array_equal(kvx.kvx_select_topk(S, k), osel.select_topk(S, k))


def test_select_topk_ties_heavy_integer_scores():
    rng = np.random.default_rng(5)
    for _ in range(200):
        lt, ls = int(rng.integers(1, 9)), int(rng.integers(1, 12))
        k = int(rng.integers(1, ls + 1))
        S = rng.integers(0, 3, size=(lt, ls)).astype(np.float64)
        assert np.array_equal(kvx.kvx_select_topk(S, k), osel.select_topk(S, k))


def test_select_topk_rejects_bad_arguments():
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_select_topk(np.zeros((3, 4)), 5)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    with pytest.raises(kvx.KvxError):
        kvx.kvx_select_topk(np.full((2, 3), np.nan), 1)


def test_mapper_params_match_paper_table_and_oracle():
    rows = [ln.split() for ln in open(os.path.join(ROOT, "tests", "golden", "mapper_sizes.txt"))
            if ln.strip() and not ln.startswith("#")]
    for name, k, lt, nkv, dh, params_b, _ in rows:
        p = kvx.kvx_mapper_params(int(lt), int(nkv), int(dh), int(k), kvx.KVX_CROSS_HEAD)
        assert round(p / 1e9, 2) == float(params_b), name
        assert p == omap.mapper_params(int(lt), int(nkv), int(dh), int(k), head_mix="cross_head")
    assert kvx.kvx_mapper_params(64, 8, 128, 4, kvx.KVX_PER_HEAD) == 2 * 64 * 8 * 512 * 128
    assert kvx.kvx_mapper_params(0, 8, 128, 4, kvx.KVX_PER_HEAD) == -1


def _cfg(**over):
    w = syn.workload("tiny_fp32")
    W, b = syn.weights(w)
    args = dict(src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k,
                theta_s=w.theta_s, theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b,
                scores=syn.selection_scores(w))
    args.update(over)
    return kvx.config_from_tensors(**args)


@pytest.mark.parametrize("field,value", [
    ("k", 0), ("k", 5), ("head_dim", 0), ("src_layers", -1), ("rope_style", 7),
    ("head_mix", 3), ("cache_dtype", 9), ("reserved", 1), ("src_rope_theta", float("nan")),
    ("tgt_rope_theta", 0.5),
])
def test_create_rejects_invalid_config_before_touching_the_device(field, value):
    cfg, keep = _cfg()
    setattr(cfg, field, value)
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_create(cfg, 0)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG, kvx.kvx_last_error()


def test_create_rejects_unsupported_head_dims():
    for hd in (63, 258):
        cfg, keep = _cfg()
        cfg.head_dim = hd
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_create(cfg, 0)
        assert e.value.status == kvx.KVX_ERR_UNSUPPORTED


def test_create_rejects_bad_selection_tables():
    w = syn.workload("tiny_fp32")
    for bad in ([[0, 0]] * 6, [[0, 4]] * 6, [[-1, 2]] * 6):
        cfg, keep = _cfg(selection=np.array(bad, dtype=np.int32), scores=None)
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_create(cfg, 0)
        assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    cfg, keep = _cfg()
    cfg.W = None
    with pytest.raises(kvx.KvxError):
        kvx.kvx_create(cfg, 0)


def test_null_arguments_are_rejected():
    L = kvx.lib()
    assert L.kvx_create(None, 0, None) == kvx.KVX_ERR_INVALID_ARG
    assert L.kvx_map(None, None, 1, 1, None, None, None) == kvx.KVX_ERR_INVALID_ARG
    assert L.kvx_destroy(None) == kvx.KVX_OK
    assert L.kvx_get_status(None, None) == kvx.KVX_ERR_INVALID_ARG
    assert L.kvx_set_kernel(None, 0) == kvx.KVX_ERR_INVALID_ARG
    assert L.kvx_get_selection(None, None) == kvx.KVX_ERR_INVALID_ARG


def test_fit_ridge_rejects_bad_arguments_before_touching_the_device():
    """kvx_fit_ridge validates everything on the host first (no GPU is needed to see it)."""
    good = dict(src_layers=4, tgt_layers=3, n_kv_heads=2, head_dim=128, k=2, theta_s=1e6, theta_t=1e6,
                lam=0.01, selection=np.array([[0, 1], [1, 2], [2, 3]], dtype=np.int32))
    buf = np.zeros(64, dtype=np.float32)          # a 16-byte aligned stand-in for device pointers
    src = kvx.kvx_src(buf.ctypes.data, buf.ctypes.data, (ctypes.c_int64 * 4)(4096, 4096, 256, 128))
    cases = [dict(head_dim=64), dict(k=5), dict(k=0), dict(lam=-1.0), dict(theta_t=1.0),
             dict(selection=np.array([[0, 4], [1, 2], [2, 3]], dtype=np.int32)),
             dict(src_layers=1)]
    for over in cases:
        a = dict(good, **over)
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_fit_ridge(a["src_layers"], a["tgt_layers"], a["n_kv_heads"], a["head_dim"], a["k"],
                              a["theta_s"], a["theta_t"], a["lam"], a["selection"], src, src, 1, 16,
                              buf.ctypes.data, buf.ctypes.data, buf.ctypes.data)
        assert e.value.status == kvx.KVX_ERR_INVALID_ARG, over
    with pytest.raises(kvx.KvxError) as e:                 # NULL output
        a = good
        kvx.kvx_fit_ridge(a["src_layers"], a["tgt_layers"], a["n_kv_heads"], a["head_dim"], a["k"],
                          a["theta_s"], a["theta_t"], a["lam"], a["selection"], src, src, 1, 16,
                          buf.ctypes.data, None, buf.ctypes.data)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_r2_probe_rejects_bad_arguments_before_touching_the_device():
    """kvx_r2_probe validates everything on the host first."""
    good = dict(src_layers=4, tgt_layers=3, n_kv_heads=2, head_dim=128, theta_s=1e6, theta_t=1e6, batch=1, T=256)
    buf = np.zeros(64, dtype=np.float64)          # an aligned stand-in for device pointers
    src = kvx.kvx_src(buf.ctypes.data, buf.ctypes.data, (ctypes.c_int64 * 4)(4096, 4096, 256, 128))
    cases = [dict(head_dim=64), dict(src_layers=0), dict(tgt_layers=0), dict(n_kv_heads=0), dict(theta_t=1.0),
             dict(theta_s=float("inf")), dict(T=128), dict(batch=0)]
    for over in cases:
        a = dict(good, **over)
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_r2_probe(a["src_layers"], a["tgt_layers"], a["n_kv_heads"], a["head_dim"], a["theta_s"],
                             a["theta_t"], src, src, a["batch"], a["T"], buf.ctypes.data, buf.ctypes.data)
        assert e.value.status == kvx.KVX_ERR_INVALID_ARG, over
    bad_stride = kvx.kvx_src(buf.ctypes.data, buf.ctypes.data, (ctypes.c_int64 * 4)(4096, 4096, 256, 100))
    with pytest.raises(kvx.KvxError):
        kvx.kvx_r2_probe(4, 3, 2, 128, 1e6, 1e6, bad_stride, src, 1, 256, buf.ctypes.data, buf.ctypes.data)
    with pytest.raises(kvx.KvxError) as e:                 # NULL scores
        kvx.kvx_r2_probe(4, 3, 2, 128, 1e6, 1e6, src, src, 1, 256, buf.ctypes.data, None)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_select_topk_device_rejects_bad_arguments_before_touching_the_device():
    buf = np.zeros(16, dtype=np.float64)
    for (lt, ls, k) in [(0, 4, 1), (3, 0, 1), (3, 4, 0), (3, 4, 5)]:
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_select_topk_device(buf.ctypes.data, lt, ls, k, buf.ctypes.data)
        assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    with pytest.raises(kvx.KvxError):
        kvx.kvx_select_topk_device(None, 3, 4, 2, buf.ctypes.data)


def test_mlp_map_rejects_bad_arguments_before_touching_the_device():
    """kvx_mlp_map validates its configuration on the host first."""
    buf = np.zeros(64, dtype=np.float64)
    p = buf.ctypes.data
    sel = np.array([[0, 1], [1, 2]], dtype=np.int32)
    good = dict(src_layers=3, tgt_layers=2, n_kv_heads=2, head_dim=128, k=2, hidden=256, theta_s=1e6, theta_t=1e6,
                selection=sel)
    src = kvx.kvx_src(p, p, (ctypes.c_int64 * 4)(4096, 4096, 256, 128))
    tgt = kvx.kvx_tgt()
    tgt.k, tgt.v = p, p
    for i, s in enumerate((4096, 4096, 256, 128)):
        tgt.stride[i] = s
    cases = [dict(head_dim=64), dict(hidden=100), dict(hidden=0), dict(k=0), dict(k=4), dict(theta_t=0.5),
             dict(selection=np.array([[0, 3], [1, 2]], dtype=np.int32)), dict(n_kv_heads=0)]
    for over in cases:
        a = dict(good, **over)
        cfg = kvx.mlp_config(a["src_layers"], a["tgt_layers"], a["n_kv_heads"], a["head_dim"], a["k"], a["hidden"],
                             a["theta_s"], a["theta_t"], a["selection"], p, p, p, p, p, p)
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_mlp_map(cfg, src, 1, 16, p, tgt)
        assert e.value.status == kvx.KVX_ERR_INVALID_ARG, over
        assert kvx.kvx_mlp_workspace_bytes(cfg, 1, 16) == -1
    cfg = kvx.mlp_config(3, 2, 2, 128, 2, 256, 1e6, 1e6, sel, p, p, None, p, p, p)   # NULL W2
    with pytest.raises(kvx.KvxError):
        kvx.kvx_mlp_map(cfg, src, 1, 16, p, tgt)
    cfg = kvx.mlp_config(3, 2, 2, 128, 2, 256, 1e6, 1e6, sel, p, p, p, p, p, p)
    assert kvx.kvx_mlp_workspace_bytes(cfg, 1, 16) > 0
    paged = kvx.kvx_tgt()
    paged.paged, paged.block_size, paged.k, paged.v = 1, 16, p, p
    for i, s in enumerate((4096, 4096, 256, 128)):
        paged.stride[i] = s
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_mlp_map(cfg, src, 1, 16, p, paged)
    assert e.value.status == kvx.KVX_ERR_UNSUPPORTED


@pytest.mark.parametrize("spec", [(0.5, 1.0, 4.0, 8192.0), (8.0, 4.0, 1.0, 8192.0), (8.0, 0.0, 4.0, 8192.0),
                                  (8.0, 1.0, 4.0, 0.0), (float("inf"), 1.0, 4.0, 8192.0)])
def test_rope_scaling_is_validated_on_the_host(spec):
    """Invalid Llama-3 scaling parameters are refused by kvx_create, kvx_fit_ridge and
    kvx_r2_probe before any device work."""
    cfg, keep = _cfg()
    rs = kvx.rope_scaling(spec)
    cfg.tgt_rope_scaling = ctypes.pointer(rs)
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_create(cfg, 0)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    buf = np.zeros(64, dtype=np.float64)
    p = buf.ctypes.data
    src = kvx.kvx_src(p, p, (ctypes.c_int64 * 4)(4096, 4096, 256, 128))
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_fit_ridge(4, 3, 2, 128, 2, 1e6, 1e6, 0.01, np.array([[0, 1], [1, 2], [2, 3]], dtype=np.int32),
                          src, src, 1, 16, p, p, p, rope_scaling=spec)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_r2_probe(4, 3, 2, 128, 1e6, 1e6, src, src, 1, 256, p, p, rope_scaling=spec)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_host_pipe_rejects_bad_arguments_before_touching_the_device():
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_host_pipe_create(None, 1, 1024)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    buf = np.zeros(64, dtype=np.float64)
    p = buf.ctypes.data
    src = kvx.kvx_src(p, p, (ctypes.c_int64 * 4)(4096, 4096, 256, 128))
    tgt = kvx.kvx_tgt()
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_map_host(None, src, 16, p, tgt)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_create_rejects_bad_rope_numerics():
    cfg, keep = _cfg()
    cfg.rope_numerics = 2
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_create(cfg, 0)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def _noalloc_mapper(sel, **over):
    """A kvx_noalloc_mapper for host-side validation only: W and b are placeholder
    16-byte aligned addresses that no check before the launch dereferences."""
    m = kvx.kvx_noalloc_mapper()
    m.src_layers, m.tgt_layers, m.n_kv_heads, m.head_dim, m.k = 4, sel.shape[0], 2, 64, sel.shape[1]
    m.rope_style = kvx.KVX_ROPE_HALF
    m.src_rope_theta = m.tgt_rope_theta = 1e4
    m.cache_dtype = m.weight_dtype = kvx.KVX_F32
    m.head_mix = kvx.KVX_PER_HEAD
    m.selection = sel.ctypes.data
    m.W, m.b = 0x10000, 0x20000
    for key, val in over.items():
        setattr(m, key, val)
    return m


@pytest.mark.parametrize("sel,over,why", [
    ([[0, 0], [1, 2]], {}, "duplicate"),
    ([[0, 3], [2, 1]], {"rope_numerics": 2}, "rope_numerics"),
    ([[0, 4], [1, 2]], {}, "outside"),
    ([[0, 1], [1, 2]], {"reserved": 1}, "reserved"),
])
def test_noalloc_rejects_bad_mapper_before_touching_the_device(sel, over, why):
    sel = np.ascontiguousarray(sel, dtype=np.int32)
    m = _noalloc_mapper(sel, **over)
    src, tgt = kvx.kvx_src(), kvx.kvx_tgt()
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_map_noalloc(m, 0, src, 1, 8, 0x30000, tgt, want_status=False)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    assert why in kvx.kvx_last_error()


def test_set_test_wait_rejects_bad_arguments():
    for args in ((None, 0, -1), (1, 10, -1), (1, 5_000_000_000, -1), (1, 0, -2), (1, 0, 2 ** 40)):
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_set_test_wait(*args)
        assert e.value.status == kvx.KVX_ERR_INVALID_ARG


def test_get_kernel_rejects_null_arguments():
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_get_kernel(None)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
