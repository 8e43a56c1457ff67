"""kvx_map_noalloc: the mapping entry point that allocates nothing.

It exists for callers that cannot let a library allocate device memory: a framework
that has reserved nearly all of the device's memory for its own pool (a library's
cudaMalloc then fails or fragments that pool), or a serving path that cannot pay the
implicit device synchronisation of cudaMalloc / cudaFree.  Its only scratch is a fixed
array inside the library that every call reuses, so each case calls it twice in a row
and requires both outputs to equal, bit for bit, what kvx_map produces with the same
SIMT kernel on a context of the same configuration; one output per case is also
checked against the float64 oracle at the tests' tolerance.  The first case's first
call carries a bad position, so its status must say so and the second call must find
that status cleared.
This file sorts last so a stop-at-first-failure run has already run everything else.
"""
import numpy as np
import pytest
import torch

from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn

from harness import check, oracle_full, oracle_rows, to_f64

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_03893_gb300 import build as kbuild
    kbuild.build()
    kvx.lib()
    torch.cuda.set_device(0)


def _bits(t):
    """Integer view of a float tensor, so NaN sentinels compare equal to themselves."""
    return t.view(torch.int16 if t.dtype == torch.bfloat16 else torch.int32)


def _simt_ctx(w, rope_style, rope_numerics):
    W, b = syn.weights(w)
    cfg, keep = kvx.config_from_tensors(
        src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k, theta_s=w.theta_s,
        theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b, scores=syn.selection_scores(w),
        rope_style=rope_style, rope_numerics=rope_numerics,
        head_mix=kvx.KVX_CROSS_HEAD if w.head_mix == "cross_head" else kvx.KVX_PER_HEAD)
    ctx = kvx.kvx_create(cfg, 0)
    kvx.kvx_set_kernel(ctx, kvx.KVX_KERNEL_SIMT)
    return ctx, kvx.kvx_get_selection(ctx, w.Lt, w.k), W, b


def _mapper(w, sel, W_dev, b_dev, rope_style=kvx.KVX_ROPE_HALF, rope_numerics=kvx.KVX_ROPE_EXACT):
    m = kvx.kvx_noalloc_mapper()
    m.src_layers, m.tgt_layers, m.n_kv_heads, m.head_dim, m.k = w.Ls, w.Lt, w.H, w.d, w.k
    m.rope_style = rope_style
    m.src_rope_theta, m.tgt_rope_theta = w.theta_s, w.theta_t
    m.cache_dtype = kvx.KVX_BF16 if w.cache_dtype == "bf16" else kvx.KVX_F32
    m.weight_dtype = kvx.dtype_code(W_dev)
    m.head_mix = kvx.KVX_CROSS_HEAD if w.head_mix == "cross_head" else kvx.KVX_PER_HEAD
    m.reserved = 0
    m.rope_numerics = rope_numerics
    m.selection = sel.ctypes.data
    m.W = W_dev.data_ptr()
    m.b = b_dev.data_ptr()
    return m


def test_noalloc_matches_kvx_map_on_two_calls_in_a_row():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=6, Lt=5, H=2, B=2, T=300, k=3)
    ctx, sel, W, b = _simt_ctx(w, kvx.KVX_ROPE_HALF, kvx.KVX_ROPE_EXACT)
    sk, sv = syn.source_cache(w, 0, device=DEV), syn.source_cache(w, 1, device=DEV)
    pos = syn.positions(w)
    pos_d = torch.from_numpy(pos).to(DEV)
    s = torch.cuda.current_stream().cuda_stream
    src = kvx.src_from_tensors(sk, sv)
    ref_k = torch.full((w.Lt, w.B, w.H, w.T, w.d), float("nan"), dtype=torch.bfloat16, device=DEV)
    ref_v = torch.full_like(ref_k, float("nan"))
    try:
        kvx.kvx_map(ctx, src, w.B, w.T, pos_d.data_ptr(), kvx.tgt_from_tensors(ref_k, ref_v), s)
        assert kvx.kvx_get_status(ctx, s) == kvx.KVX_OK
    finally:
        kvx.kvx_destroy(ctx)
    sel = np.ascontiguousarray(sel, dtype=np.int32)
    W_dev, b_dev = W.to(DEV).contiguous(), b.float().to(DEV).contiguous()
    m = _mapper(w, sel, W_dev, b_dev)

    # call 1: one bad position -> DEVICE_BOUNDS, that token left untouched, the rest
    # bit-identical to kvx_map
    bad = pos.copy()
    bad[1, 7] = -5
    bad_d = torch.from_numpy(bad).to(DEV)
    k1, v1 = torch.full_like(ref_k, float("nan")), torch.full_like(ref_v, float("nan"))
    st1 = kvx.kvx_map_noalloc(m, 0, src, w.B, w.T, bad_d.data_ptr(), kvx.tgt_from_tensors(k1, v1), s)
    assert st1 == kvx.KVX_ERR_DEVICE_BOUNDS
    assert torch.isnan(k1[:, 1, :, 7]).all() and torch.isnan(v1[:, 1, :, 7]).all()
    k1[:, 1, :, 7] = ref_k[:, 1, :, 7]
    v1[:, 1, :, 7] = ref_v[:, 1, :, 7]
    assert torch.equal(_bits(k1), _bits(ref_k)) and torch.equal(_bits(v1), _bits(ref_v))

    # call 2: valid positions; the status left by call 1 must have been cleared
    k2, v2 = torch.full_like(ref_k, float("nan")), torch.full_like(ref_v, float("nan"))
    st2 = kvx.kvx_map_noalloc(m, 0, src, w.B, w.T, pos_d.data_ptr(), kvx.tgt_from_tensors(k2, v2), s)
    assert st2 == kvx.KVX_OK
    assert torch.equal(_bits(k2), _bits(ref_k)) and torch.equal(_bits(v2), _bits(ref_v))
    rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b)
    ok, ratio, rms, nbad = check(w, [to_f64(k2), to_f64(v2)], [rk, rv], [ak, av])
    assert ok, "call 2 vs oracle: %d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)


CASES = {
    # fp32 caches and fp32 W (the tiny workload's precision)
    "fp32": dict(name="tiny_fp32", over=dict(T=150)),
    # the paper's feature layout: every KV head of the selected layers feeds every target head
    "cross_head": dict(name="qwen3_14b_32b_b8x1024_k4_xhead", over=dict(Ls=4, Lt=3, H=2, B=1, T=130, k=2)),
    # RoPE pairs (2i, 2i+1)
    "interleaved": dict(name="qwen3_14b_32b_b8x1024_k4", over=dict(Ls=5, Lt=4, H=2, B=1, T=140, k=2),
                        rope_style=kvx.KVX_ROPE_INTERLEAVED),
    # the Hugging Face bf16 forward's RoPE rounding (checked against kvx_map only: its
    # oracle comparison, with the bound that numerics needs, is in the map tests)
    "hf_numerics": dict(name="qwen3_14b_32b_b8x1024_k4", over=dict(Ls=5, Lt=4, H=2, B=2, T=90, k=2),
                        rope_numerics=kvx.KVX_ROPE_HF),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_noalloc_variants_contiguous(case):
    c = CASES[case]
    w = syn.workload(c["name"], **c["over"])
    style = c.get("rope_style", kvx.KVX_ROPE_HALF)
    numerics = c.get("rope_numerics", kvx.KVX_ROPE_EXACT)
    ctx, sel, W, b = _simt_ctx(w, style, numerics)
    dt = w.torch_dtype()
    sk, sv = syn.source_cache(w, 0, device=DEV), syn.source_cache(w, 1, device=DEV)
    pos = syn.positions(w) + (7001 if numerics == kvx.KVX_ROPE_HF else 0)
    pos = np.ascontiguousarray(pos, dtype=np.int32)
    pos_d = torch.from_numpy(pos).to(DEV)
    s = torch.cuda.current_stream().cuda_stream
    src = kvx.src_from_tensors(sk, sv)

    def fresh():
        t = torch.full((w.Lt, w.B, w.H, w.T, w.d), float("nan"), dtype=dt, device=DEV)
        return t, torch.full_like(t, float("nan"))

    ref_k, ref_v = fresh()
    try:
        kvx.kvx_map(ctx, src, w.B, w.T, pos_d.data_ptr(), kvx.tgt_from_tensors(ref_k, ref_v), s)
        assert kvx.kvx_get_status(ctx, s) == kvx.KVX_OK
    finally:
        kvx.kvx_destroy(ctx)
    sel = np.ascontiguousarray(sel, dtype=np.int32)
    W_dev, b_dev = W.to(DEV).contiguous(), b.float().to(DEV).contiguous()
    m = _mapper(w, sel, W_dev, b_dev, style, numerics)
    outs = []
    for _ in range(2):
        k_, v_ = fresh()
        st = kvx.kvx_map_noalloc(m, 0, src, w.B, w.T, pos_d.data_ptr(), kvx.tgt_from_tensors(k_, v_), s)
        assert st == kvx.KVX_OK
        assert torch.equal(_bits(k_), _bits(ref_k)) and torch.equal(_bits(v_), _bits(ref_v))
        outs.append((k_, v_))
    if numerics == kvx.KVX_ROPE_EXACT:
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b,
                                     style="interleaved" if style == kvx.KVX_ROPE_INTERLEAVED else "half")
        ok, ratio, rms, nbad = check(w, [to_f64(outs[1][0]), to_f64(outs[1][1])], [rk, rv], [ak, av])
        assert ok, "%s vs oracle: %d elements out of tolerance (worst %.3g x bound)" % (case, nbad, ratio)


def test_noalloc_paged_target_two_calls():
    """A paged target through the block table, two turns in a row into fresh pools: every
    slot bit-identical to kvx_map's (sentinels included), every mapped row within the
    oracle's tolerance."""
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", Ls=5, Lt=3, H=2, B=3, T=37, k=2,
                     len_range=(3, 70))
    ctx, sel, W, b = _simt_ctx(w, kvx.KVX_ROPE_HALF, kvx.KVX_ROPE_EXACT)
    L0 = syn.initial_lengths(w)
    s = torch.cuda.current_stream().cuda_stream
    sel = np.ascontiguousarray(sel, dtype=np.int32)
    W_dev, b_dev = W.to(DEV).contiguous(), b.float().to(DEV).contiguous()
    m = _mapper(w, sel, W_dev, b_dev)
    try:
        for turn in (0, 1):
            pos = syn.positions(w, turn, L0)
            table, n_blocks = syn.block_table(w, pos, turn)
            tbl, pos_d = torch.from_numpy(table).to(DEV), torch.from_numpy(pos).to(DEV)
            sk = syn.source_cache(w, 0, device=DEV, turn=turn)
            sv = syn.source_cache(w, 1, device=DEV, turn=turn)
            src = kvx.src_from_tensors(sk, sv)

            def pools():
                p = torch.empty((w.Lt, n_blocks, w.H, w.block_size, w.d), dtype=torch.bfloat16, device=DEV)
                p.view(torch.int16).fill_(0x7FBF)
                q = torch.empty_like(p)
                q.view(torch.int16).fill_(0x7FBF)
                return p, q

            ref_k, ref_v = pools()
            kvx.kvx_map(ctx, src, w.B, w.T, pos_d.data_ptr(),
                        kvx.tgt_paged_from_tensors(ref_k, ref_v, tbl, w.block_size), s)
            assert kvx.kvx_get_status(ctx, s) == kvx.KVX_OK
            pk, pv = pools()
            st = kvx.kvx_map_noalloc(m, 0, src, w.B, w.T, pos_d.data_ptr(),
                                     kvx.tgt_paged_from_tensors(pk, pv, tbl, w.block_size), s)
            assert st == kvx.KVX_OK
            assert torch.equal(_bits(pk), _bits(ref_k)) and torch.equal(_bits(pv), _bits(ref_v))
            rows = np.array([(bb, t) for bb in range(w.B) for t in range(w.T)], dtype=np.int64)
            rk, rv, ak, av = oracle_rows(w, rows, pos, sel, W, b, turn=turn)
            p = pos[rows[:, 0], rows[:, 1]]
            blk = table[rows[:, 0], p // w.block_size].astype(np.int64)
            slot = (p % w.block_size).astype(np.int64)
            gk = to_f64(pk[:, blk, :, slot].permute(1, 2, 0, 3))
            gv = to_f64(pv[:, blk, :, slot].permute(1, 2, 0, 3))
            ok, ratio, rms, nbad = check(w, [gk, gv], [rk, rv], [ak, av])
            assert ok, "paged turn %d vs oracle: %d out of tolerance (worst %.3g)" % (turn, nbad, ratio)
    finally:
        kvx.kvx_destroy(ctx)


def test_noalloc_rejects_oversized_selection():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=6, Lt=5000, H=1, B=1, T=8, k=4)
    sel = np.zeros((w.Lt, w.k), dtype=np.int32)
    sel[:] = np.arange(4)
    dummy = torch.zeros(64, dtype=torch.bfloat16, device=DEV)
    m = _mapper(w, sel, dummy, dummy.float())
    t = torch.zeros((1, 1, 1, 8, 128), dtype=torch.bfloat16, device=DEV)
    pos = torch.zeros((1, 8), dtype=torch.int32, device=DEV)
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_map_noalloc(m, 0, kvx.src_from_tensors(t, t), 1, 8, pos.data_ptr(),
                            kvx.tgt_from_tensors(t, t))
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    assert "KVX_NOALLOC_MAX_SELECTION" in kvx.kvx_last_error()
