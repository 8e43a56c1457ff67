"""kvx_map_noalloc: the mapping entry point that allocates nothing.

It exists for callers that cannot let a library allocate device memory (a framework
that has reserved the device's memory for its own pool, or a serving path that cannot
pay cudaMalloc's implicit synchronisation).  Its only scratch is a fixed array inside
the library that every call reuses, so the test calls it twice in a row: the first call
carries a bad position (its status must say so), the second a valid one (the status the
first call left behind must have been cleared), and both outputs must match the
existing entry point (kvx_map with the same SIMT kernel) within the tests' tolerance.
This file sorts last so a stop-at-first-failure run has already run everything else.
"""
import numpy as np
import pytest
import torch

from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn

from harness import check, make_ctx, run_contiguous, to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_03893_gb300 import build as kbuild
    kbuild.build()
    kvx.lib()
    torch.cuda.set_device(0)


def _mapper(w, sel, W_dev, b_dev):
    m = kvx.kvx_noalloc_mapper()
    m.src_layers, m.tgt_layers, m.n_kv_heads, m.head_dim, m.k = w.Ls, w.Lt, w.H, w.d, w.k
    m.rope_style = kvx.KVX_ROPE_HALF
    m.src_rope_theta, m.tgt_rope_theta = w.theta_s, w.theta_t
    m.cache_dtype = kvx.KVX_BF16 if w.cache_dtype == "bf16" else kvx.KVX_F32
    m.weight_dtype = kvx.dtype_code(W_dev)
    m.head_mix, m.reserved = kvx.KVX_PER_HEAD, 0
    m.selection = sel.ctypes.data
    m.W = W_dev.data_ptr()
    m.b = b_dev.data_ptr()
    return m


def test_noalloc_matches_kvx_map_on_two_calls_in_a_row():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=6, Lt=5, H=2, B=2, T=300, k=3)
    dev = torch.device("cuda:0")
    ctx, sel, W, b = make_ctx(w, kernel=kvx.KVX_KERNEL_SIMT)
    try:
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        ref_k, ref_v, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
    finally:
        kvx.kvx_destroy(ctx)
    sel = np.ascontiguousarray(sel, dtype=np.int32)
    W_dev = W.to(dev).contiguous()
    b_dev = b.float().to(dev).contiguous()
    m = _mapper(w, sel, W_dev, b_dev)
    s = torch.cuda.current_stream().cuda_stream
    src = kvx.src_from_tensors(sk, sv)

    # call 1: one bad position -> DEVICE_BOUNDS, that token left untouched
    bad = pos.copy()
    bad[1, 7] = -5
    bad_d = torch.from_numpy(bad).to(dev)
    k1 = torch.full_like(ref_k, float("nan"))
    v1 = torch.full_like(ref_v, float("nan"))
    st1 = kvx.kvx_map_noalloc(m, 0, src, w.B, w.T, bad_d.data_ptr(), kvx.tgt_from_tensors(k1, v1), s)
    assert st1 == kvx.KVX_ERR_DEVICE_BOUNDS
    mask = torch.ones(w.B, w.T, dtype=torch.bool, device=dev)
    mask[1, 7] = False

    def rows(x):  # [L][B][H][T][d] -> [L][tokens kept][H][d]
        return x.permute(0, 1, 3, 2, 4)[:, mask]

    assert torch.isnan(k1[:, 1, :, 7]).all()
    ok, ratio, rms, nbad = check(w, [to_f64(rows(k1)), to_f64(rows(v1))],
                                 [to_f64(rows(ref_k)), to_f64(rows(ref_v))])
    assert ok, "call 1: %d elements out of tolerance" % nbad

    # call 2: valid positions; the status left by call 1 must have been cleared
    pos_d = torch.from_numpy(pos).to(dev)
    k2 = torch.full_like(ref_k, float("nan"))
    v2 = torch.full_like(ref_v, float("nan"))
    st2 = kvx.kvx_map_noalloc(m, 0, src, w.B, w.T, pos_d.data_ptr(), kvx.tgt_from_tensors(k2, v2), s)
    assert st2 == kvx.KVX_OK
    ok, ratio, rms, nbad = check(w, [to_f64(k2), to_f64(v2)], [to_f64(ref_k), to_f64(ref_v)])
    assert ok, "call 2: %d elements out of tolerance" % nbad


def test_noalloc_rejects_oversized_selection():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=6, Lt=5000, H=1, B=1, T=8, k=4)
    sel = np.zeros((w.Lt, w.k), dtype=np.int32)
    sel[:] = np.arange(4)
    dummy = torch.zeros(64, dtype=torch.bfloat16, device="cuda:0")
    m = _mapper(w, sel, dummy, dummy.float())
    t = torch.zeros((1, 1, 1, 8, 128), dtype=torch.bfloat16, device="cuda:0")
    pos = torch.zeros((1, 8), dtype=torch.int32, device="cuda:0")
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_map_noalloc(m, 0, kvx.src_from_tensors(t, t), 1, 8, pos.data_ptr(),
                            kvx.tgt_from_tensors(t, t))
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    assert "KVX_NOALLOC_MAX_SELECTION" in kvx.kvx_last_error()
