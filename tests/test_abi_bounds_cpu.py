"""Host checks of the fit, probe, MLP and no-alloc entry points and of the Llama-3 RoPE
scaling parameters, at every boundary (CPU).

Each bound is checked from both sides, one field at a time with the others valid.  A
rejection returns before any device work, so those cases run anywhere.  Acceptance is
seen without a device where the ABI offers a way: kvx_map_noalloc and kvx_mlp_map return
KVX_OK for an empty batch right after their checks, and the probe's and MLP's
workspace-size queries are host-only.  The remaining acceptances (a call that passes
every check) go on to the device; they are checked only where no GPU is present, where
the first CUDA call fails with KVX_ERR_CUDA, because on a GPU they would launch kernels
on the placeholder pointers these tests use."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_03893_gb300 import build as kbuild
from paper_2608_03893_gb300 import kvx

INV = kvx.KVX_ERR_INVALID_ARG
device_free = pytest.mark.skipif(torch.cuda.is_available(),
                                 reason="an accepted call would launch kernels on placeholder pointers")

_BUF = np.zeros(1 << 16, dtype=np.uint8)
BASE = (_BUF.ctypes.data + 255) // 256 * 256     # a 256-byte aligned placeholder address


@pytest.fixture(scope="module", autouse=True)
def built():
    kbuild.build()
    kvx.lib()


def _sel(rows):
    return np.ascontiguousarray(rows, dtype=np.int32)


def _src(**over):
    s = kvx.kvx_src(BASE, BASE + 4096, (ctypes.c_int64 * 4)(1 << 20, 1 << 16, 1 << 12, 128))
    for key, val in over.items():
        if key.startswith("stride"):
            s.stride[int(key[-1])] = val
        else:
            setattr(s, key, val)
    return s


def _tgt(**over):
    t = kvx.kvx_tgt()
    t.k, t.v = BASE + 8192, BASE + 12288
    for i, v in enumerate((1 << 20, 1 << 16, 1 << 12, 128)):
        t.stride[i] = v
    for key, val in over.items():
        if key.startswith("stride"):
            t.stride[int(key[-1])] = val
        else:
            setattr(t, key, val)
    return t


# ----------------------------------------------------------------- RoPE scaling ------

SCALING_OK = (8.0, 1.0, 4.0, 8192.0)
SCALING_BAD = [(0.999, 1.0, 4.0, 8192.0), (np.inf, 1.0, 4.0, 8192.0), (np.nan, 1.0, 4.0, 8192.0),
               (8.0, 0.0, 4.0, 8192.0), (8.0, np.nan, 4.0, 8192.0), (8.0, 1.0, 1.0, 8192.0),
               (8.0, 1.0, np.inf, 8192.0), (8.0, 1.0, np.nan, 8192.0), (8.0, 1.0, 4.0, 0.0),
               (8.0, 1.0, 4.0, np.inf), (8.0, 1.0, 4.0, np.nan)]
SCALING_EDGE_OK = [(1.0, 1.0, 4.0, 8192.0), (8.0, 1e-9, 4.0, 8192.0), (8.0, 1.0, 1.0 + 1e-12, 8192.0),
                   (8.0, 1.0, 4.0, 1e-9)]


# ----------------------------------------------------------------- no-alloc map ------

def _mapper(sel=None, **over):
    sel = _sel([[0, 2], [1, 3], [0, 3]]) if sel is None else sel
    m = kvx.kvx_noalloc_mapper()
    m.src_layers, m.tgt_layers, m.n_kv_heads, m.head_dim, m.k = 4, sel.shape[0], 2, 64, sel.shape[1]
    m.rope_style, m.cache_dtype, m.weight_dtype, m.head_mix = kvx.KVX_ROPE_HALF, kvx.KVX_F32, kvx.KVX_F32, 0
    m.src_rope_theta = m.tgt_rope_theta = 1e4
    m.selection, m.W, m.b = sel.ctypes.data, BASE, BASE + 1024
    for key, val in over.items():
        setattr(m, key, val)
    m._sel = sel
    return m


def _noalloc(m, batch=0, T=8, src=None, tgt=None, pos=BASE + 16384, use_src=True, use_tgt=True):
    src = _src() if src is None else src
    tgt = _tgt() if tgt is None else tgt
    return kvx.lib().kvx_map_noalloc(ctypes.byref(m) if m is not None else None, 0,
                                     ctypes.byref(src) if use_src else None, batch, T, pos,
                                     ctypes.byref(tgt) if use_tgt else None, None, None)


def _with_scaling(m, which, spec):
    rs = kvx.kvx_rope_scaling(*spec)
    setattr(m, which, ctypes.pointer(rs))
    m._rs = rs
    return m


def test_rope_scaling_bounds():
    for which in ("src_rope_scaling", "tgt_rope_scaling"):
        assert _noalloc(_with_scaling(_mapper(), which, SCALING_OK)) == kvx.KVX_OK
        for spec in SCALING_EDGE_OK:
            assert _noalloc(_with_scaling(_mapper(), which, spec)) == kvx.KVX_OK, (which, spec)
        for spec in SCALING_BAD:
            assert _noalloc(_with_scaling(_mapper(), which, spec)) == INV, (which, spec)


def test_noalloc_config_bounds():
    assert _noalloc(_mapper()) == kvx.KVX_OK                         # an empty batch after the checks
    assert _noalloc(_mapper(), batch=2, T=0) == kvx.KVX_OK
    for field in ("src_layers", "tgt_layers", "n_kv_heads", "head_dim"):
        assert _noalloc(_mapper(**{field: 0})) == INV, field
    for hd, want in ((63, INV), (2, kvx.KVX_OK), (256, kvx.KVX_OK), (258, INV)):
        assert _noalloc(_mapper(head_dim=hd)) == want, hd
    assert _noalloc(_mapper(sel=_sel([[0, 1, 2, 3]] * 3))) == kvx.KVX_OK       # k = L_s
    assert _noalloc(_mapper(sel=_sel([[3]] * 3))) == kvx.KVX_OK                # k = 1
    m = _mapper(sel=_sel([[0, 1, 2, 3]] * 3))
    m.k = 0
    assert _noalloc(m) == INV
    m = _mapper(sel=_sel([[0, 1, 2, 3, 0]] * 3))                               # k = L_s + 1
    assert _noalloc(m) == INV
    # L_t k = 16384 fits the selection array, one more does not
    assert _noalloc(_mapper(sel=_sel(np.tile([[0, 1]], (8192, 1))))) == kvx.KVX_OK
    assert _noalloc(_mapper(sel=_sel(np.tile([[1]], (16385, 1))))) == INV
    for field, good, bad in (("rope_style", (0, 1), 2), ("cache_dtype", (0, 1), 2), ("weight_dtype", (0, 1), 2),
                             ("head_mix", (0, 1), 2), ("rope_numerics", (0, 1), 2), ("reserved", (0,), 1)):
        for v in good:
            assert _noalloc(_mapper(**{field: v})) == kvx.KVX_OK, (field, v)
        assert _noalloc(_mapper(**{field: bad})) == INV, field
    for field in ("src_rope_theta", "tgt_rope_theta"):
        assert _noalloc(_mapper(**{field: 1.0 + 1e-9})) == kvx.KVX_OK, field
        for bad in (1.0, np.inf, np.nan):
            assert _noalloc(_mapper(**{field: bad})) == INV, (field, bad)
    for field in ("selection", "W", "b"):
        assert _noalloc(_mapper(**{field: None})) == INV, field
    for field in ("W", "b"):
        assert _noalloc(_mapper(**{field: BASE + 8})) == INV, field
        assert _noalloc(_mapper(**{field: BASE + 16})) == kvx.KVX_OK, field


def test_noalloc_selection_bounds():
    assert _noalloc(_mapper(sel=_sel([[0, 3], [1, 2], [0, 3]]))) == kvx.KVX_OK
    for bad in ([[0, 4], [1, 2], [0, 3]], [[-1, 2], [1, 2], [0, 3]], [[0, 2], [1, 2], [0, 4]]):
        assert _noalloc(_mapper(sel=_sel(bad))) == INV, bad
    for row in ([1, 2, 1], [2, 1, 1], [1, 1, 2]):              # a repeat anywhere in a row
        assert _noalloc(_mapper(sel=_sel([[0, 1, 2], [0, 1, 3], row]))) == INV, row


def test_noalloc_call_bounds():
    m = _mapper()
    assert _noalloc(None) == INV
    assert _noalloc(m, use_src=False) == INV
    assert _noalloc(m, use_tgt=False) == INV
    assert _noalloc(m, batch=-1) == INV
    assert _noalloc(m, batch=1, T=-1) == INV
    for field in ("k", "v"):
        assert _noalloc(m, batch=1, src=_src(**{field: None})) == INV, field
        assert _noalloc(m, batch=1, tgt=_tgt(**{field: None})) == INV, field
        assert _noalloc(m, batch=1, src=_src(**{field: BASE + 8})) == INV, field
        assert _noalloc(m, batch=1, tgt=_tgt(**{field: BASE + 8})) == INV, field
    assert _noalloc(m, batch=1, pos=None) == INV
    assert _noalloc(m, batch=1, pos=BASE + 2) == INV
    for i in range(4):
        for bad in (-8, 4):
            assert _noalloc(m, batch=1, src=_src(**{"stride%d" % i: bad})) == INV, (i, bad)
            assert _noalloc(m, batch=1, tgt=_tgt(**{"stride%d" % i: bad})) == INV, (i, bad)
    assert _noalloc(m, batch=1, src=_src(stride3=56)) == INV          # token stride < head_dim 64
    assert _noalloc(m, batch=1, tgt=_tgt(stride3=56)) == INV
    assert _noalloc(m, batch=1, tgt=_tgt(paged=2)) == INV
    paged = dict(paged=1, block_size=16, block_table=BASE + 20480, max_blocks_per_seq=4, n_blocks=8)
    for key, bad in (("block_size", 0), ("block_table", None), ("block_table", BASE + 20482),
                     ("max_blocks_per_seq", 0), ("n_blocks", 0)):
        assert _noalloc(m, batch=1, tgt=_tgt(**dict(paged, **{key: bad}))) == INV, key


@device_free
def test_noalloc_call_accepted_reaches_the_device():
    m = _mapper()
    assert _noalloc(m, batch=1) == kvx.KVX_ERR_CUDA
    assert _noalloc(m, batch=1, src=_src(stride3=64), tgt=_tgt(stride3=64), pos=BASE + 4) == kvx.KVX_ERR_CUDA
    paged = dict(paged=1, block_size=16, block_table=BASE + 20480, max_blocks_per_seq=4, n_blocks=8)
    assert _noalloc(m, batch=1, tgt=_tgt(**paged)) == kvx.KVX_ERR_CUDA
    for i in range(3):
        assert _noalloc(m, batch=1, src=_src(**{"stride%d" % i: 0}), tgt=_tgt(**{"stride%d" % i: 0})) == \
            kvx.KVX_ERR_CUDA, i


# ----------------------------------------------------------------- ridge fit ---------

def _fit_cfg(sel=None, **over):
    sel = _sel([[0, 1], [1, 2], [2, 3]]) if sel is None else sel
    c = kvx.kvx_fit_config()
    c.src_layers, c.tgt_layers, c.n_kv_heads, c.head_dim, c.k = 4, sel.shape[0], 2, 128, sel.shape[1]
    c.src_rope_theta = c.tgt_rope_theta = 1e6
    c.lambda_ = 0.01
    c.selection = sel.ctypes.data
    c.head_mix = kvx.KVX_PER_HEAD
    for key, val in over.items():
        setattr(c, key, val)
    c._sel = sel
    return c


def _fit(c, batch=1, T=16, src=None, tgt=None, pos=BASE + 16384, W=BASE + 32768, b=BASE + 49152,
         use_src=True, use_tgt=True):
    src = _src() if src is None else src
    tgt = _src() if tgt is None else tgt
    return kvx.lib().kvx_fit_ridge(ctypes.byref(c) if c is not None else None,
                                   ctypes.byref(src) if use_src else None, ctypes.byref(tgt) if use_tgt else None,
                                   batch, T, pos, W, b, None)


def test_fit_config_rejections():
    assert _fit(None) == INV
    for hd in (127, 129, 64):
        assert _fit(_fit_cfg(head_dim=hd)) == INV, hd
    assert _fit(_fit_cfg(head_mix=2)) == INV
    assert _fit(_fit_cfg(sel=_sel([[0, 1, 2, 3, 0]] * 3), src_layers=5)) == INV        # per head: k <= 4
    c = _fit_cfg()
    c.k = 0
    assert _fit(c) == INV
    # cross-head: k n_kv 128 <= 16384
    assert _fit(_fit_cfg(sel=_sel(np.tile(np.arange(17), (2, 1))), src_layers=17, n_kv_heads=8,
                         head_mix=kvx.KVX_CROSS_HEAD)) == INV
    c = _fit_cfg(head_mix=kvx.KVX_CROSS_HEAD)
    c.k = 0
    assert _fit(c) == INV
    for field in ("src_layers", "tgt_layers", "n_kv_heads"):
        assert _fit(_fit_cfg(**{field: 0})) == INV, field
    assert _fit(_fit_cfg(src_layers=1)) == INV                                      # k = 2 > L_s
    for field, bad in (("lambda_", -1e-12), ("lambda_", np.nan), ("src_rope_theta", 1.0),
                       ("tgt_rope_theta", 1.0), ("src_rope_theta", np.nan), ("tgt_rope_theta", np.nan)):
        assert _fit(_fit_cfg(**{field: bad})) == INV, (field, bad)
    assert _fit(_fit_cfg(selection=None)) == INV
    for bad in ([[0, 4], [1, 2], [2, 3]], [[0, 1], [1, 2], [-1, 3]], [[0, 1], [1, 2], [2, 4]]):
        assert _fit(_fit_cfg(sel=_sel(bad))) == INV, bad
    assert _fit(_fit_cfg(workspace=None, workspace_bytes=1024)) == INV
    assert _fit(_fit_cfg(workspace=BASE + 16, workspace_bytes=1024)) == INV              # not 256-aligned
    assert _fit(_fit_cfg(rope_numerics=2)) == INV
    for which in ("src_rope_scaling", "tgt_rope_scaling"):
        c = _fit_cfg()
        rs = kvx.kvx_rope_scaling(0.5, 1.0, 4.0, 8192.0)
        setattr(c, which, ctypes.pointer(rs))
        assert _fit(c) == INV, which


def test_fit_call_rejections():
    c = _fit_cfg()
    assert _fit(c, use_src=False) == INV
    assert _fit(c, use_tgt=False) == INV
    for key in ("pos", "W", "b"):
        assert _fit(c, **{key: None}) == INV, key
    assert _fit(c, batch=0) == INV and _fit(c, T=0) == INV
    for which in ("src", "tgt"):
        for field, bad in (("k", None), ("v", None), ("k", BASE + 8), ("v", BASE + 8)):
            assert _fit(c, **{which: _src(**{field: bad})}) == INV, (which, field, bad)
        for i in range(4):
            for bad in (-8, 4):
                assert _fit(c, **{which: _src(**{"stride%d" % i: bad})}) == INV, (which, i, bad)
        assert _fit(c, **{which: _src(stride3=120)}) == INV                          # token stride < 128
    assert _fit(c, pos=BASE + 2) == INV
    assert _fit(c, W=BASE + 8) == INV and _fit(c, b=BASE + 8) == INV


@device_free
def test_fit_accepted_reaches_the_device():
    # the first accepted value of every bound, one at a time
    cases = [dict(), dict(lambda_=0.0), dict(src_rope_theta=1.0 + 1e-9), dict(tgt_rope_theta=1.0 + 1e-9),
             dict(workspace=BASE, workspace_bytes=1024), dict(rope_numerics=1),
             dict(sel=_sel([[0, 1, 2, 3]] * 3)), dict(sel=_sel([[3]] * 3)),
             dict(sel=_sel(np.tile(np.arange(16), (2, 1))), src_layers=16, n_kv_heads=8,
                  head_mix=kvx.KVX_CROSS_HEAD)]
    cases += [dict(sel=_sel([[0]]), src_layers=1), dict(n_kv_heads=1),
              dict(sel=_sel([[0, 1]] * 1)), dict(sel=_sel([[2]] * 3), head_mix=kvx.KVX_CROSS_HEAD)]
    for over in cases:
        assert _fit(_fit_cfg(**over)) == kvx.KVX_ERR_CUDA, over
    assert _fit(_fit_cfg(), src=_src(stride3=128), pos=BASE + 4, W=BASE + 16, b=BASE + 16) == kvx.KVX_ERR_CUDA
    assert _fit(_fit_cfg(), batch=1, T=1) == kvx.KVX_ERR_CUDA
    for i in range(3):                                   # a zero stride repeats a layer, batch or head
        assert _fit(_fit_cfg(), src=_src(**{"stride%d" % i: 0}), tgt=_src(**{"stride%d" % i: 0})) == \
            kvx.KVX_ERR_CUDA, i


# ----------------------------------------------------------------- R^2 probe ---------

def _probe_cfg(**over):
    c = kvx.kvx_probe_config(4, 3, 2, 128, 1e6, 1e6, None, 0)
    for key, val in over.items():
        setattr(c, key, val)
    return c


def _probe_ws(c, batch=1, T=256):
    return kvx.lib().kvx_r2_probe_workspace_bytes(ctypes.byref(c), batch, T)


def _probe(c, batch=1, T=256, src=None, tgt=None, pos=BASE + 16384, scores=BASE + 32768, r2=BASE + 40960,
           use_src=True, use_tgt=True):
    src = _src() if src is None else src
    tgt = _src() if tgt is None else tgt
    return kvx.lib().kvx_r2_probe(ctypes.byref(c) if c is not None else None,
                                  ctypes.byref(src) if use_src else None, ctypes.byref(tgt) if use_tgt else None,
                                  batch, T, pos, scores, r2, None)


def test_probe_config_bounds():
    assert _probe_ws(_probe_cfg()) > 0
    for over in (dict(head_dim=127), dict(head_dim=129), dict(src_layers=0), dict(tgt_layers=0),
                 dict(n_kv_heads=0), dict(src_rope_theta=1.0), dict(tgt_rope_theta=1.0),
                 dict(src_rope_theta=np.inf), dict(tgt_rope_theta=np.inf), dict(src_rope_theta=np.nan),
                 dict(workspace=None, workspace_bytes=1), dict(workspace=BASE + 128, workspace_bytes=1),
                 dict(rope_numerics=2)):
        assert _probe_ws(_probe_cfg(**over)) == -1, over
        assert _probe(_probe_cfg(**over)) == INV, over
    for over in (dict(src_rope_theta=1.0 + 1e-9), dict(tgt_rope_theta=1.0 + 1e-9), dict(rope_numerics=1),
                 dict(workspace=BASE, workspace_bytes=1), dict(src_layers=1, tgt_layers=1, n_kv_heads=1)):
        assert _probe_ws(_probe_cfg(**over)) > 0, over
    for which in ("src_rope_scaling", "tgt_rope_scaling"):
        c = _probe_cfg()
        rs = kvx.kvx_rope_scaling(8.0, 0.0, 4.0, 8192.0)
        setattr(c, which, ctypes.pointer(rs))
        assert _probe_ws(c) == -1 and _probe(c) == INV, which
    assert _probe_ws(_probe_cfg(), batch=0) == -1 and _probe_ws(_probe_cfg(), T=0) == -1


def test_probe_call_rejections():
    c = _probe_cfg()
    assert _probe(None) == INV
    assert _probe(c, use_src=False) == INV and _probe(c, use_tgt=False) == INV
    assert _probe(c, pos=None) == INV and _probe(c, scores=None) == INV
    assert _probe(c, batch=0) == INV and _probe(c, T=0) == INV
    assert _probe(c, T=128) == INV and _probe(c, batch=2, T=64) == INV      # 128 tokens or fewer
    for which in ("src", "tgt"):
        for field, bad in (("k", None), ("v", None), ("k", BASE + 8), ("v", BASE + 8)):
            assert _probe(c, **{which: _src(**{field: bad})}) == INV, (which, field, bad)
        for i in range(4):
            for bad in (-8, 4):
                assert _probe(c, **{which: _src(**{"stride%d" % i: bad})}) == INV, (which, i, bad)
        assert _probe(c, **{which: _src(stride3=120)}) == INV
    assert _probe(c, pos=BASE + 2) == INV
    assert _probe(c, scores=BASE + 4) == INV and _probe(c, r2=BASE + 4) == INV


@device_free
def test_probe_accepted_reaches_the_device():
    c = _probe_cfg()
    assert _probe(c, T=129) == kvx.KVX_ERR_CUDA
    assert _probe(c, r2=None) == kvx.KVX_ERR_CUDA
    assert _probe(c, src=_src(stride3=128), pos=BASE + 4, scores=BASE + 8, r2=BASE + 8) == kvx.KVX_ERR_CUDA
    assert _probe(c, batch=129, T=1) == kvx.KVX_ERR_CUDA
    for i in range(3):
        assert _probe(c, src=_src(**{"stride%d" % i: 0}), tgt=_src(**{"stride%d" % i: 0})) == kvx.KVX_ERR_CUDA, i


# ----------------------------------------------------------------- MLP mapper --------

def _mlp_cfg(sel=None, **over):
    sel = _sel([[0, 1], [1, 2]]) if sel is None else sel
    p = [BASE + 1024 * i for i in range(6)]
    c = kvx.mlp_config(3, sel.shape[0], 2, 128, sel.shape[1], 256, 1e6, 1e6, sel, *p)
    for key, val in over.items():
        setattr(c, key, val)
    return c


def _mlp_ws(c):
    return kvx.lib().kvx_mlp_workspace_bytes(ctypes.byref(c), 1, 16)


def _mlp(c, batch=1, T=16, src=None, tgt=None, pos=BASE + 16384, use_src=True, use_tgt=True):
    src = _src() if src is None else src
    tgt = _tgt() if tgt is None else tgt
    return kvx.lib().kvx_mlp_map(ctypes.byref(c) if c is not None else None, ctypes.byref(src) if use_src else None,
                                 batch, T, pos, ctypes.byref(tgt) if use_tgt else None, None)


def test_mlp_config_bounds():
    assert _mlp_ws(_mlp_cfg()) > 0 and _mlp(_mlp_cfg(), batch=0) == kvx.KVX_OK
    bad = [dict(head_dim=127), dict(head_dim=129), dict(src_layers=0), dict(tgt_layers=0), dict(n_kv_heads=0),
           dict(hidden=0), dict(hidden=255), dict(hidden=257), dict(hidden=65792), dict(src_rope_theta=1.0),
           dict(tgt_rope_theta=1.0), dict(src_rope_theta=np.inf), dict(tgt_rope_theta=np.nan),
           dict(selection=None), dict(workspace=None, workspace_bytes=1), dict(workspace=BASE + 128, workspace_bytes=1),
           dict(rope_numerics=2)]
    bad += [{w: None} for w in ("W1", "b1", "W2", "b2", "W3", "b3")]
    bad += [{w: BASE + 8} for w in ("W1", "b1", "W2", "b2", "W3", "b3")]
    for over in bad:
        assert _mlp_ws(_mlp_cfg(**over)) == -1, over
        assert _mlp(_mlp_cfg(**over)) == INV, over
    good = [dict(hidden=512), dict(hidden=65536), dict(src_rope_theta=1.0 + 1e-9), dict(rope_numerics=1),
            dict(n_kv_heads=1), dict(sel=_sel([[0]] * 2), src_layers=1), dict(sel=_sel([[1, 2]]), tgt_layers=1),
            dict(workspace=BASE, workspace_bytes=1), dict(sel=_sel([[0, 1, 2]] * 2)), dict(sel=_sel([[2]] * 2))]
    good += [{w: BASE + 16} for w in ("W1", "b1", "W2", "b2", "W3", "b3")]
    for over in good:
        assert _mlp_ws(_mlp_cfg(**over)) > 0, over
        assert _mlp(_mlp_cfg(**over), batch=0) == kvx.KVX_OK, over
    c = _mlp_cfg(sel=_sel([[0, 1, 2]] * 2))
    c.k = 0
    assert _mlp_ws(c) == -1
    c = _mlp_cfg(sel=_sel([[0, 1, 2, 0]] * 2))                      # k = L_s + 1
    assert _mlp_ws(c) == -1
    for rows in ([[0, 3], [1, 2]], [[0, 1], [-1, 2]], [[0, 1], [1, 3]]):
        assert _mlp_ws(_mlp_cfg(sel=_sel(rows))) == -1, rows
    # weight rows: L_t 2 n_kv hidden <= 2^30 - 1
    assert _mlp_ws(_mlp_cfg(sel=_sel([[0]]), n_kv_heads=8191, hidden=65536)) > 0
    assert _mlp_ws(_mlp_cfg(sel=_sel([[0]]), n_kv_heads=8192, hidden=65536)) == -1
    for which in ("src_rope_scaling", "tgt_rope_scaling"):
        c = _mlp_cfg()
        rs = kvx.kvx_rope_scaling(8.0, 1.0, 4.0, 0.0)
        setattr(c, which, ctypes.pointer(rs))
        assert _mlp_ws(c) == -1, which


def test_mlp_call_bounds():
    c = _mlp_cfg()
    assert _mlp(None) == INV
    assert _mlp(c, use_src=False) == INV and _mlp(c, use_tgt=False) == INV and _mlp(c, pos=None) == INV
    assert _mlp(c, batch=-1) == INV and _mlp(c, T=-1) == INV
    assert _mlp(c, T=0) == kvx.KVX_OK
    for field in ("k", "v"):
        assert _mlp(c, src=_src(**{field: None})) == INV, field
        assert _mlp(c, tgt=_tgt(**{field: None})) == INV, field
        assert _mlp(c, src=_src(**{field: BASE + 8})) == INV, field
        assert _mlp(c, tgt=_tgt(**{field: BASE + 8})) == INV, field
    assert _mlp(c, tgt=_tgt(paged=1)) == kvx.KVX_ERR_UNSUPPORTED
    for i in range(4):
        for bad in (-8, 4):
            assert _mlp(c, src=_src(**{"stride%d" % i: bad})) == INV, (i, bad)
            assert _mlp(c, tgt=_tgt(**{"stride%d" % i: bad})) == INV, (i, bad)
    assert _mlp(c, src=_src(stride3=120)) == INV and _mlp(c, tgt=_tgt(stride3=120)) == INV
    assert _mlp(c, pos=BASE + 2) == INV


@device_free
def test_mlp_accepted_reaches_the_device():
    c = _mlp_cfg()
    assert _mlp(c) == kvx.KVX_ERR_CUDA
    assert _mlp(c, src=_src(stride3=128), tgt=_tgt(stride3=128), pos=BASE + 4) == kvx.KVX_ERR_CUDA
    for i in range(3):
        assert _mlp(c, src=_src(**{"stride%d" % i: 0}), tgt=_tgt(**{"stride%d" % i: 0})) == kvx.KVX_ERR_CUDA, i
