"""The Python binding's marshalling on CPU tensors (no GPU): every struct field it fills
from a tensor or an argument, and the errors it raises before calling the library."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_03893_gb300 import build as kbuild
from paper_2608_03893_gb300 import kvx


@pytest.fixture(scope="module", autouse=True)
def built():
    kbuild.build()
    kvx.lib()


def _read_i32(addr, n):
    return np.ctypeslib.as_array((ctypes.c_int32 * n).from_address(addr)).copy()


def _read_f64(addr, n):
    return np.ctypeslib.as_array((ctypes.c_double * n).from_address(addr)).copy()


def test_src_and_tgt_from_tensors():
    base_k = torch.zeros(3, 2, 4, 10, 64)
    base_v = torch.zeros(3, 2, 4, 10, 64)
    k, v = base_k[:, :, :, 2:9], base_v[:, :, :, 2:9]             # a strided view: T = 7 of 10
    s = kvx.src_from_tensors(k, v)
    assert (s.k, s.v) == (k.data_ptr(), v.data_ptr())
    assert list(s.stride) == list(k.stride()[:4]) == [2 * 4 * 10 * 64, 4 * 10 * 64, 10 * 64, 64]
    t = kvx.tgt_from_tensors(k, v)
    assert (t.paged, t.block_size, t.k, t.v) == (0, 0, k.data_ptr(), v.data_ptr())
    assert list(t.stride) == list(k.stride()[:4])
    assert not t.block_table and (t.max_blocks_per_seq, t.n_blocks) == (0, 0)
    for bad in ((k, torch.zeros(3, 2, 4, 7, 64)),                   # same shape, other strides
                (k, v[:2]),                                        # different shapes
                (k.transpose(3, 4), v.transpose(3, 4))):           # head_dim not contiguous
        with pytest.raises(ValueError):
            kvx.src_from_tensors(*bad)
        with pytest.raises(ValueError):
            kvx.tgt_from_tensors(*bad)


def test_paged_target_from_tensors():
    pk = torch.zeros(5, 9, 2, 16, 64)                              # [L][n_blocks][H][block][d]
    pv = torch.zeros(5, 9, 2, 16, 64)
    table = torch.zeros(3, 7, dtype=torch.int32)
    t = kvx.tgt_paged_from_tensors(pk, pv, table, 16)
    assert (t.paged, t.block_size, t.k, t.v) == (1, 16, pk.data_ptr(), pv.data_ptr())
    assert list(t.stride) == list(pk.stride()[:4])
    assert (t.block_table, t.max_blocks_per_seq, t.n_blocks) == (table.data_ptr(), 7, 9)
    with pytest.raises(ValueError):
        kvx.tgt_paged_from_tensors(pk, pv, table, 8)               # slot axis != block_size
    with pytest.raises(ValueError):
        kvx.tgt_paged_from_tensors(pk, pv[:, :8], table, 16)


def test_config_from_tensors_fills_every_field():
    W = torch.randn(4, 2, 3, 128, 64)
    b = torch.randn(4, 2, 3, 64, dtype=torch.float64)              # converted to W's dtype
    sel = [[0, 2], [1, 2], [0, 1], [2, 3]]
    cfg, keep = kvx.config_from_tensors(src_layers=5, tgt_layers=4, n_kv_heads=3, head_dim=64, k=2,
                                        theta_s=1e4, theta_t=5e5, cache_dtype="bf16", W=W, b=b,
                                        selection=sel, rope_style=kvx.KVX_ROPE_INTERLEAVED,
                                        head_mix=kvx.KVX_PER_HEAD, rope_scaling=(8.0, 1.0, 4.0, 8192.0),
                                        rope_numerics=kvx.KVX_ROPE_HF)
    assert (cfg.src_layers, cfg.tgt_layers, cfg.n_kv_heads, cfg.head_dim, cfg.k) == (5, 4, 3, 64, 2)
    assert (cfg.src_rope_theta, cfg.tgt_rope_theta) == (1e4, 5e5)
    assert (cfg.rope_style, cfg.head_mix, cfg.reserved, cfg.rope_numerics) == (1, 0, 0, 1)
    assert (cfg.cache_dtype, cfg.weight_dtype) == (kvx.KVX_BF16, kvx.KVX_F32)
    assert np.array_equal(_read_i32(cfg.selection, 8), np.array(sel).ravel())
    assert not cfg.selection_scores
    got_W = np.ctypeslib.as_array((ctypes.c_float * W.numel()).from_address(cfg.W))
    assert np.array_equal(got_W, W.numpy().ravel())
    got_b = np.ctypeslib.as_array((ctypes.c_float * b.numel()).from_address(cfg.b))
    assert np.array_equal(got_b, b.float().numpy().ravel())
    for p in (cfg.src_rope_scaling, cfg.tgt_rope_scaling):
        assert (p.contents.factor, p.contents.low_freq_factor, p.contents.high_freq_factor,
                p.contents.original_max_position) == (8.0, 1.0, 4.0, 8192.0)
    # scores instead of a selection; bf16 weights; an integer cache dtype; no bias
    S = np.random.default_rng(0).uniform(size=(4, 5))
    cfg, keep = kvx.config_from_tensors(src_layers=5, tgt_layers=4, n_kv_heads=3, head_dim=64, k=2,
                                        theta_s=1e4, theta_t=1e4, cache_dtype=kvx.KVX_F32,
                                        W=W.to(torch.bfloat16), scores=S)
    assert (cfg.cache_dtype, cfg.weight_dtype) == (kvx.KVX_F32, kvx.KVX_BF16)
    assert not cfg.selection and not cfg.b and np.array_equal(_read_f64(cfg.selection_scores, 20), S.ravel())
    assert not cfg.src_rope_scaling and not cfg.tgt_rope_scaling and cfg.rope_numerics == 0
    with pytest.raises(ValueError):
        kvx.config_from_tensors(src_layers=5, tgt_layers=4, n_kv_heads=3, head_dim=64, k=2, theta_s=1e4,
                                theta_t=1e4, cache_dtype="f32", W=W)
    with pytest.raises(TypeError):
        kvx.dtype_code(torch.zeros(1, dtype=torch.float16))


def test_mlp_config_and_scaling_helpers():
    sel = np.array([[0, 1], [1, 2]])
    cfg = kvx.mlp_config(3, 2, 2, 128, 2, 256, 1e6, 5e5, sel, 16, 32, 48, 64, 80, 96, workspace_ptr=256,
                         workspace_bytes=4096, rope_scaling=(8.0, 1.0, 4.0, 8192.0), rope_numerics=1)
    assert (cfg.src_layers, cfg.tgt_layers, cfg.n_kv_heads, cfg.head_dim, cfg.k, cfg.hidden) == (3, 2, 2, 128, 2, 256)
    assert (cfg.src_rope_theta, cfg.tgt_rope_theta) == (1e6, 5e5)
    assert (cfg.W1, cfg.b1, cfg.W2, cfg.b2, cfg.W3, cfg.b3) == (16, 32, 48, 64, 80, 96)
    assert (cfg.workspace, cfg.workspace_bytes, cfg.rope_numerics) == (256, 4096, 1)
    assert np.array_equal(_read_i32(cfg.selection, 4), sel.ravel())
    assert cfg.src_rope_scaling.contents.factor == 8.0 and cfg.tgt_rope_scaling.contents.factor == 8.0
    assert kvx.rope_scaling(None) is None and not kvx._scaling_ptr(None)


def test_errors_carry_the_status_and_the_library_message():
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_select_topk(np.zeros((2, 3)), 4)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    assert "kvx_select_topk" in str(e.value) and "KVX_ERR_INVALID_ARG" in str(e.value)
    assert "k must be in [1, src_layers]" in str(e.value)
    assert kvx.kvx_mapper_params(64, 8, 128, 4) == 2 * 64 * 8 * 4 * 128 * 128
    assert kvx.kvx_mapper_params(64, 8, 128, 4, kvx.KVX_CROSS_HEAD) == 2 * 64 * 8 * 4 * 8 * 128 * 128


def test_a_missing_library_fails_loudly(monkeypatch, tmp_path):
    # no fallback: every entry point goes through lib(), which raises without libkvx.so
    monkeypatch.setattr(kvx, "_lib", None)
    monkeypatch.setattr(kvx, "LIB_PATH", str(tmp_path / "libkvx.so"))
    with pytest.raises(RuntimeError, match="libkvx.so not found"):
        kvx.lib()
    with pytest.raises(RuntimeError):
        kvx.kvx_select_topk(np.zeros((2, 3)), 1)
    with pytest.raises(RuntimeError):
        kvx.kvx_mapper_params(64, 8, 128, 4)
