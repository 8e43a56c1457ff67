"""GPU parity: the CUDA path (through the C ABI) against the float64 oracle on the same
seeded inputs.  Small shapes are compared in full; the full-size workloads are compared
on sampled token rows (all layers, heads, K and V of each sampled token) plus checks
that hold at any size (every row written, untouched paged slots keep their sentinel)."""
import numpy as np
import pytest
import torch

from oracle import mapper as omap
from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn

from harness import (check, make_ctx, oracle_full, oracle_rows, run_contiguous, sample_rows,
                     to_f64)

pytestmark = pytest.mark.gpu

KERNELS = {"simt": kvx.KVX_KERNEL_SIMT, "tc": kvx.KVX_KERNEL_TCGEN05}


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_03893_gb300 import build as kbuild
    kbuild.build()
    kvx.lib()
    torch.cuda.set_device(0)


def _kernel_or_skip(w, kernel):
    ctx, sel, W, b = make_ctx(w)
    try:
        if kernel == kvx.KVX_KERNEL_TCGEN05:
            try:
                kvx.kvx_set_kernel(ctx, kernel)
            except kvx.KvxError as e:
                pytest.fail("tensor-core kernel unavailable for a bf16 d=128 shape: %s" % e)
    finally:
        kvx.kvx_destroy(ctx)


def _small(name, kernel, **over):
    w = syn.workload(name, **over)
    ctx, sel, W, b = make_ctx(w, kernel=kernel)
    try:
        dev = torch.device("cuda:0")
        sk = syn.source_cache(w, 0, device=dev)
        sv = syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        tk, tv, status = run_contiguous(ctx, w, sk, sv, pos)
        assert status == kvx.KVX_OK
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b)
        ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
        assert ok, "%s: %d elements out of tolerance (worst %.3g x bound)" % (name, nbad, ratio)
        return ratio
    finally:
        kvx.kvx_destroy(ctx)


# ----------------------------------------------------------------- small, full -----

def test_tiny_fp32_full():
    _small("tiny_fp32", kvx.KVX_KERNEL_AUTO)


@pytest.mark.parametrize("kname", ["simt", "tc"])
@pytest.mark.parametrize("over", [
    dict(Ls=6, Lt=5, H=2, B=2, T=300, k=3),                # ragged tail, B > 1
    dict(Ls=3, Lt=4, H=1, B=1, T=1, k=1),                  # one token
    dict(Ls=5, Lt=7, H=2, B=3, T=129, k=2, theta_t=5e5),   # different thetas, 1-row tail
    dict(Ls=9, Lt=6, H=3, B=1, T=640, k=4),                # several tiles
    dict(Ls=8, Lt=9, H=2, B=1, T=256, k=4, scores="uniform"),  # random selection, reloads
    dict(Ls=10, Lt=5, H=2, B=1, T=200, k=5),               # beyond the tensor-core kernel: SIMT
])
def test_bf16_small_full(kname, over):
    name = "qwen3_14b_32b_b8x1024_k4"
    if kname == "tc":
        _kernel_or_skip(syn.workload(name, **over), KERNELS[kname])
    _small(name, KERNELS[kname], **over)


@pytest.mark.parametrize("over", [
    dict(Ls=10, Lt=5, H=2, B=1, T=200, k=5),                 # k = 5, one ragged tile
    dict(Ls=12, Lt=4, H=4, B=2, T=300, k=8),                 # k = 8, B > 1
    dict(Ls=9, Lt=3, H=2, B=1, T=257, k=8, scores="uniform", theta_t=5e5),
])
def test_per_head_beyond_four_layers_on_tensor_cores(over):
    """Per-head mappers with k > 4 (more selected layers than the per-head kernel keeps in
    tensor memory) run on the cross-head tensor-core kernel with W widened by zeros outside
    each head's rows: AUTO picks it, every element matches the oracle, and repeated launches
    agree."""
    name = "qwen3_14b_32b_b8x1024_k4"
    w = syn.workload(name, **over)
    ctx, sel, W, b = make_ctx(w)
    try:
        assert kvx.kvx_get_kernel(ctx) == 3 and kvx.kvx_get_kernel(ctx, paged=True) == 3
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b)
        first = None
        for rep in range(3):
            tk, tv, status = run_contiguous(ctx, w, sk, sv, pos)
            assert status == kvx.KVX_OK
            ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
            assert ok, "%d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
            if first is None:
                first = (tk.clone(), tv.clone())
            else:
                assert torch.equal(tk, first[0]) and torch.equal(tv, first[1])
        kvx.kvx_set_kernel(ctx, kvx.KVX_KERNEL_SIMT)
        assert kvx.kvx_get_kernel(ctx) == 1
    finally:
        kvx.kvx_destroy(ctx)


@pytest.mark.parametrize("over", [
    dict(Ls=6, Lt=5, H=2, B=2, T=300, k=3),
    dict(Ls=9, Lt=6, H=3, B=1, T=640, k=4),
    dict(Ls=8, Lt=9, H=2, B=1, T=256, k=4, scores="uniform"),
])
def test_tc_small_repeated(over):
    """Eight launches of one small shape (one work unit per CTA, so every role starts cold):
    a race between the kernel's roles shows up as a launch that differs from the oracle."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", **over)
    _kernel_or_skip(w, kvx.KVX_KERNEL_TCGEN05)
    ctx, sel, W, b = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b)
        for rep in range(8):
            tk, tv, status = run_contiguous(ctx, w, sk, sv, pos)
            assert status == kvx.KVX_OK
            ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
            assert ok, "launch %d: %d elements out of tolerance (worst %.3g x bound)" % (rep, nbad, ratio)
    finally:
        kvx.kvx_destroy(ctx)


def test_interleaved_pairs_simt():
    w = syn.workload("tiny_fp32", T=100, B=2)
    ctx, sel, W, b = make_ctx(w, rope_style=kvx.KVX_ROPE_INTERLEAVED)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w) + 7
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b, style="interleaved")
        assert check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])[0]
    finally:
        kvx.kvx_destroy(ctx)


# ------------------------------------------------------ interleaved RoPE pairs -----

@pytest.mark.parametrize("name,over,weights,expect", [
    ("qwen3_14b_32b_b8x1024_k4", dict(Ls=6, Lt=4, H=2, B=2, T=300, k=3, theta_t=5e5), "bf16", 2),
    ("qwen3_14b_32b_b8x1024_k4", dict(Ls=6, Lt=5, H=2, B=1, T=260, k=4, scores="uniform"), "f32", 2),
    ("qwen3_14b_32b_b8x1024_k4", dict(Ls=9, Lt=3, H=2, B=1, T=200, k=6), "bf16", 3),   # k > 4: widened W
    ("qwen3_14b_32b_t32768_k4_xhead", dict(Ls=4, Lt=3, H=2, B=2, T=150, k=2), "bf16", 3),
])
def test_interleaved_pairs_tensor_cores(name, over, weights, expect):
    """Interleaved RoPE pairs (2i, 2i+1) on the per-head (2) and cross-head (3) tensor-core
    kernels, bf16 and fp32 (hi + lo) weights: every output element of two launches against
    the float64 oracle in the interleaved style, at positions past 10^4; the half-split
    oracle's keys fail the same bound (the test sees the pairing)."""
    w = syn.workload(name, **over)
    Wb, b = syn.weights(w)
    W = Wb
    if weights == "f32":
        g = torch.Generator().manual_seed(7)
        W = (Wb.float() * (1.0 + 2.0 ** -9 * torch.rand(Wb.shape, generator=g))).contiguous()
    ctx, sel, _, _ = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05, W=W, b=b, rope_style=kvx.KVX_ROPE_INTERLEAVED)
    try:
        assert kvx.kvx_get_kernel(ctx) == expect
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w) + 10007
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b, style="interleaved")
        for rep in range(2):
            tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
            assert st == kvx.KVX_OK
            ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
            assert ok, "launch %d: %d elements out of tolerance (worst %.3g x bound)" % (rep, nbad, ratio)
        hk, _, hak, _ = oracle_full(w, sk, sv, pos, sel, W, b, style="half")
        assert not check(w, [to_f64(tk)], [hk], [hak])[0]
    finally:
        kvx.kvx_destroy(ctx)


@pytest.mark.parametrize("kname,name", [("simt", "qwen3_14b_32b_b8x1024_k4"), ("tc", "qwen3_14b_32b_b8x1024_k4"),
                                        ("tc", "qwen3_14b_32b_t32768_k4_xhead")])
def test_interleaved_pairs_hf_numerics(kname, name):
    """Interleaved pairs with KVX_ROPE_HF (fp32 angle, bf16 cos / sin, every product and sum
    rounded) on the SIMT, per-head and cross-head kernels: values within the bound of the
    HF oracle, keys within 4 bf16 steps of their pair's magnitude and at least 90 % of them
    bit-equal to it, far more than agree with the exact-RoPE oracle."""
    w = syn.workload(name, Ls=5, Lt=3, H=2, B=2, T=180, k=2, theta_t=5e5)
    W, b = syn.weights(w)
    mix = kvx.KVX_CROSS_HEAD if w.head_mix == "cross_head" else kvx.KVX_PER_HEAD
    cfg, keep = kvx.config_from_tensors(
        src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k, theta_s=w.theta_s,
        theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b, scores=syn.selection_scores(w),
        rope_style=kvx.KVX_ROPE_INTERLEAVED, head_mix=mix, rope_numerics=kvx.KVX_ROPE_HF)
    ctx = kvx.kvx_create(cfg, 0)
    try:
        kvx.kvx_set_kernel(ctx, KERNELS[kname])
        sel = kvx.kvx_get_selection(ctx, w.Lt, w.k)
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w) + np.array([[20011], [31007]], dtype=np.int32)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        sk64, sv64 = to_f64(sk), to_f64(sv)
        common = dict(mode="bf16fwd", style="interleaved", head_mix=w.head_mix)
        rk, rv = omap.map_cache(sk64, sv64, pos, sel, to_f64(W), to_f64(b), w.theta_s, w.theta_t,
                                rope_numerics="hf", **common)
        ek, _ = omap.map_cache(sk64, sv64, pos, sel, to_f64(W), to_f64(b), w.theta_s, w.theta_t, **common)
        gk, gv = to_f64(tk), to_f64(tv)
        ok, ratio, rms, nbad = check(w, [gv], [rv])
        assert ok, "values: %d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
        mag = np.repeat(np.abs(rk[..., 0::2]) + np.abs(rk[..., 1::2]), 2, axis=-1)
        assert np.all(np.abs(gk - rk) <= 2.0 ** -6 * mag + 1e-3 * rms)
        from oracle import bf16 as obf16
        same_hf, same_exact = np.mean(gk == rk), np.mean(gk == obf16.round_to_bf16_value(ek))
        assert same_hf >= 0.9 and same_hf > same_exact + 0.1, (same_hf, same_exact)
    finally:
        kvx.kvx_destroy(ctx)


def test_cross_head_simt():
    w = syn.workload("tiny_fp32", T=64)
    Wc = torch.from_numpy((np.random.default_rng(3).standard_normal(
        (w.Lt, 2, w.H, w.k * w.H * w.d, w.d)) / np.sqrt(w.k * w.H * w.d)).astype(np.float32))
    _, b = syn.weights(w)
    scores = syn.selection_scores(w)
    cfg, keep = kvx.config_from_tensors(
        src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k,
        theta_s=w.theta_s, theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=Wc, b=b,
        scores=scores, head_mix=kvx.KVX_CROSS_HEAD)
    ctx = kvx.kvx_create(cfg, 0)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        sel = kvx.kvx_get_selection(ctx, w.Lt, w.k)
        rk, rv = omap.map_cache(to_f64(sk), to_f64(sv), pos, sel, to_f64(Wc), to_f64(b),
                                w.theta_s, w.theta_t, mode="exact", head_mix="cross_head")
        assert check(w, [to_f64(tk), to_f64(tv)], [rk, rv])[0]
    finally:
        kvx.kvx_destroy(ctx)


@pytest.mark.parametrize("kname", ["simt", "tc"])
def test_identity_map_is_bit_exact(kname):
    """k = 1, W = I, b = 0, equal thetas: V comes back bit for bit; K too at position 0
    (the strip and re-rotation are exact identities there)."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=3, Lt=3, H=2, B=1, T=200, k=1)
    W = torch.zeros((w.Lt, 2, w.H, w.d, w.d), dtype=torch.float32)
    W[:, :, :] = torch.eye(w.d)
    W = W.to(torch.bfloat16)
    sel = np.array([[2], [0], [1]], dtype=np.int32)
    ctx, sel_out, _, _ = make_ctx(w, kernel=KERNELS[kname], selection=sel, W=W, b=None)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = np.zeros((1, w.T), dtype=np.int32)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        for l in range(w.Lt):
            assert torch.equal(tv[l], sv[sel[l, 0]])
            assert torch.equal(tk[l], sk[sel[l, 0]])
    finally:
        kvx.kvx_destroy(ctx)


def test_empty_and_errors():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=3, Lt=2, H=2, B=1, T=16, k=2)
    ctx, sel, W, b = make_ctx(w)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        tk = torch.zeros((w.Lt, w.B, w.H, w.T, w.d), dtype=torch.bfloat16, device=dev)
        tv = torch.zeros_like(tk)
        pos = torch.zeros((1, w.T), dtype=torch.int32, device=dev)
        src, tgt = kvx.src_from_tensors(sk, sv), kvx.tgt_from_tensors(tk, tv)
        s = torch.cuda.current_stream().cuda_stream
        kvx.kvx_map(ctx, src, 0, w.T, pos.data_ptr(), tgt, s)       # empty batch: no-op
        kvx.kvx_map(ctx, src, 1, 0, pos.data_ptr(), tgt, s)         # no tokens: no-op
        assert kvx.kvx_get_status(ctx, s) == kvx.KVX_OK
        assert torch.count_nonzero(tk) == 0
        # misaligned pointer -> INVALID_ARG, nothing launched
        bad = kvx.src_from_tensors(sk, sv)
        bad.k = sk.data_ptr() + 2
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_map(ctx, bad, 1, w.T, pos.data_ptr(), tgt, s)
        assert e.value.status == kvx.KVX_ERR_INVALID_ARG
        # negative position -> device status DEVICE_BOUNDS, that row not written
        pos[0, 5] = -3
        kvx.kvx_map(ctx, src, 1, w.T, pos.data_ptr(), tgt, s)
        assert kvx.kvx_get_status(ctx, s) == kvx.KVX_ERR_DEVICE_BOUNDS
        assert kvx.kvx_get_status(ctx, s) == kvx.KVX_OK              # reset after read
        assert torch.count_nonzero(tk[:, 0, :, 5]) == 0
        assert torch.count_nonzero(tk[:, 0, :, 4]) > 0
    finally:
        kvx.kvx_destroy(ctx)


def test_generator_cpu_gpu_identical():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=2, B=2, T=300)
    g = syn.source_cache(w, 0, device=torch.device("cuda:0")).cpu()
    c = syn.source_cache(w, 0, device="cpu")
    assert torch.equal(g.view(torch.int16), c.view(torch.int16))


# ------------------------------------------------------------ full size, sampled -----

FULL = ["qwen3_14b_32b_b8x1024_k4", "qwen3_14b_32b_t32768_k1", "qwen3_14b_32b_t32768_k2",
        "qwen3_14b_32b_t32768_k4", "llama31_8b_70b_b4x8192_k3", "llama31_70b_8b_b4x8192_k3"]


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled(name):
    w = syn.workload(name)
    ctx, sel, W, b = make_ctx(w)            # AUTO: the kernel the bench times
    dev = torch.device("cuda:0")
    try:
        sk = syn.source_cache(w, 0, device=dev)
        sv = syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        del sk, sv
        assert not torch.isnan(tk).any() and not torch.isnan(tv).any(), "unwritten rows"
        rows = sample_rows(w, 48)
        rk, rv, ak, av = oracle_rows(w, rows, pos, sel, W, b)
        gk = to_f64(tk[:, rows[:, 0], :, rows[:, 1]].permute(1, 2, 0, 3))
        gv = to_f64(tv[:, rows[:, 0], :, rows[:, 1]].permute(1, 2, 0, 3))
        ok, ratio, rms, nbad = check(w, [gk, gv], [rk, rv], [ak, av])
        assert ok, "%s: %d sampled elements out of tolerance (worst %.3g x bound)" % (name, nbad, ratio)
    finally:
        kvx.kvx_destroy(ctx)
        torch.cuda.empty_cache()


# ----------------------------------------------------------------------- paged -----

def _paged_run(w, turn, L0, ctx):
    dev = torch.device("cuda:0")
    pos = syn.positions(w, turn, L0)
    table, n_blocks = syn.block_table(w, pos, turn)
    pool_k = torch.empty((w.Lt, n_blocks, w.H, w.block_size, w.d), dtype=torch.bfloat16, device=dev)
    pool_k.view(torch.int16).fill_(0x7FBF)   # a NaN pattern the map never writes
    pool_v = torch.empty_like(pool_k)
    pool_v.view(torch.int16).fill_(0x7FBF)
    sk = syn.source_cache(w, 0, device=dev, turn=turn)
    sv = syn.source_cache(w, 1, device=dev, turn=turn)
    tbl = torch.from_numpy(table).to(dev)
    posd = torch.from_numpy(pos).to(dev)
    s = torch.cuda.current_stream().cuda_stream
    kvx.kvx_map(ctx, kvx.src_from_tensors(sk, sv), w.B, w.T, posd.data_ptr(),
                kvx.tgt_paged_from_tensors(pool_k, pool_v, tbl, w.block_size), s)
    st = kvx.kvx_get_status(ctx, s)
    return pool_k, pool_v, pos, table, n_blocks, st


def _check_paged(w, ctx, sel, W, b, turn, L0, rows):
    pool_k, pool_v, pos, table, n_blocks, st = _paged_run(w, turn, L0, ctx)
    assert st == kvx.KVX_OK
    # every slot of a mapped position is written; every other slot keeps the sentinel
    written = torch.zeros((n_blocks, w.block_size), dtype=torch.bool)
    for bb in range(w.B):
        blk = torch.from_numpy(table[bb, pos[bb] // w.block_size].astype(np.int64))
        slot = torch.from_numpy((pos[bb] % w.block_size).astype(np.int64))
        written[blk, slot] = True
    written = written.to(pool_k.device)
    for pool in (pool_k, pool_v):
        sent = pool.view(torch.int16) == 0x7FBF                     # [Lt][nb][H][bs][d]
        all_sent = sent.all(dim=-1).all(dim=2).all(dim=0)            # [nb][bs]
        none_sent = (~sent).all(dim=-1).all(dim=2).all(dim=0)
        assert torch.equal(all_sent, ~written), "a slot outside the mapped tokens was touched"
        assert torch.equal(none_sent, written), "a mapped slot was not fully written"
    rk, rv, ak, av = oracle_rows(w, rows, pos, sel, W, b, turn=turn)
    p = pos[rows[:, 0], rows[:, 1]]
    blk = table[rows[:, 0], p // w.block_size].astype(np.int64)
    slot = (p % w.block_size).astype(np.int64)
    gk = to_f64(pool_k[:, blk, :, slot].permute(1, 2, 0, 3))
    gv = to_f64(pool_v[:, blk, :, slot].permute(1, 2, 0, 3))
    ok, ratio, rms, nbad = check(w, [gk, gv], [rk, rv], [ak, av])
    assert ok, "paged turn %d: %d out of tolerance (worst %.3g)" % (turn, nbad, ratio)


@pytest.mark.parametrize("kname", ["simt", "tc"])
def test_paged_small_full(kname):
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", Ls=5, Lt=3, H=2, B=3, T=37, k=2,
                     len_range=(3, 70))
    if kname == "tc":
        _kernel_or_skip(w, KERNELS[kname])
    ctx, sel, W, b = make_ctx(w, kernel=KERNELS[kname])
    try:
        L0 = syn.initial_lengths(w)
        rows = np.array([(bb, t) for bb in range(w.B) for t in range(w.T)], dtype=np.int64)
        for turn in (0, 1):
            _check_paged(w, ctx, sel, W, b, turn, L0, rows)
        if kname == "tc":   # repeated launches: a race between roles shows up as a differing launch
            for rep in range(6):
                _check_paged(w, ctx, sel, W, b, rep % 2, L0, rows)
    finally:
        kvx.kvx_destroy(ctx)


@pytest.mark.parametrize("head_mix,expect", [("per_head", 2), ("cross_head", 3)])
def test_paged_interleaved_tensor_cores(head_mix, expect):
    """Interleaved RoPE pairs into a paged target on the tensor-core kernels (per-head and
    cross-head): every slot of two turns against the interleaved oracle, untouched slots
    keep their sentinel."""
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", Ls=5, Lt=3, H=2, B=3, T=150, k=2,
                     len_range=(3, 70), head_mix=head_mix, rope_style="interleaved")
    ctx, sel, W, b = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05)
    try:
        assert kvx.kvx_get_kernel(ctx, paged=True) == expect
        L0 = syn.initial_lengths(w)
        rows = np.array([(bb, t) for bb in range(w.B) for t in range(w.T)], dtype=np.int64)
        for turn in (0, 1):
            _check_paged(w, ctx, sel, W, b, turn, L0, rows)
    finally:
        kvx.kvx_destroy(ctx)


@pytest.mark.parametrize("turn", [0, 7])
def test_paged_full_size_sampled(turn):
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4")
    ctx, sel, W, b = make_ctx(w)
    try:
        L0 = syn.initial_lengths(w)
        _check_paged(w, ctx, sel, W, b, turn, L0, sample_rows(w, 40, seed=turn))
    finally:
        kvx.kvx_destroy(ctx)
        torch.cuda.empty_cache()


def test_paged_bad_block_is_reported_and_skipped():
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", Ls=3, Lt=2, H=2, B=2, T=20, k=2,
                     len_range=(5, 9))
    ctx, sel, W, b = make_ctx(w)
    dev = torch.device("cuda:0")
    try:
        L0 = syn.initial_lengths(w)
        pos = syn.positions(w, 0, L0)
        table, n_blocks = syn.block_table(w, pos, 0)
        table[1, pos[1, 0] // w.block_size] = n_blocks + 5        # outside the pool
        pool_k = torch.zeros((w.Lt, n_blocks, w.H, w.block_size, w.d), dtype=torch.bfloat16, device=dev)
        pool_v = torch.zeros_like(pool_k)
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        tbl, posd = torch.from_numpy(table).to(dev), torch.from_numpy(pos).to(dev)
        s = torch.cuda.current_stream().cuda_stream
        kvx.kvx_map(ctx, kvx.src_from_tensors(sk, sv), w.B, w.T, posd.data_ptr(),
                    kvx.tgt_paged_from_tensors(pool_k, pool_v, tbl, w.block_size), s)
        assert kvx.kvx_get_status(ctx, s) == kvx.KVX_ERR_DEVICE_BOUNDS
        # sequence 0 was mapped normally
        blk0 = int(table[0, pos[0, 0] // w.block_size])
        assert torch.count_nonzero(pool_k[:, blk0]) > 0
    finally:
        kvx.kvx_destroy(ctx)


def test_incremental_turns_equal_one_shot():
    """Per-token independence (the map is per token): mapping turn 0 then turn 1 into a
    contiguous cache equals mapping both turns' tokens at once."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=6, Lt=4, H=2, B=1, T=256, k=2)
    ctx, sel, W, b = make_ctx(w)
    dev = torch.device("cuda:0")
    try:
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        full_k, full_v, st = run_contiguous(ctx, w, sk, sv, pos)
        tk = torch.zeros_like(full_k)
        tv = torch.zeros_like(full_v)
        for lo, hi in ((0, 100), (100, 256)):
            tgt = (tk[:, :, :, lo:hi], tv[:, :, :, lo:hi])
            run_contiguous(ctx, w, sk[:, :, :, lo:hi], sv[:, :, :, lo:hi], pos[:, lo:hi], tgt=tgt)
        assert torch.equal(tk, full_k) and torch.equal(tv, full_v)
    finally:
        kvx.kvx_destroy(ctx)


@pytest.mark.parametrize("kname", ["simt", "tc"])
def test_target_layouts_bit_identical(kname):
    """Target caches in other strided layouts ([L][H][B][T][d] and [L][B][T][H][d] viewed as
    (L, B, H, T, d)) get the same bits as the contiguous one: the tensor-core kernel writes
    those through its direct-store path, the contiguous one through per-warp TMA stores."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=6, Lt=5, H=2, B=2, T=300, k=3)
    _kernel_or_skip(w, KERNELS[kname])
    ctx, sel, W, b = make_ctx(w, kernel=KERNELS[kname])
    dev = torch.device("cuda:0")
    try:
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        ref_k, ref_v, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        shapes = {"lhbtd": (w.Lt, w.H, w.B, w.T, w.d), "lbthd": (w.Lt, w.B, w.T, w.H, w.d)}
        perms = {"lhbtd": (0, 2, 1, 3, 4), "lbthd": (0, 1, 3, 2, 4)}
        for name, shape in shapes.items():
            bk = torch.full(shape, float("nan"), dtype=sk.dtype, device=dev)
            bv = torch.full_like(bk, float("nan"))
            tk, tv = bk.permute(*perms[name]), bv.permute(*perms[name])
            assert tk.shape == ref_k.shape
            _, _, st = run_contiguous(ctx, w, sk, sv, pos, tgt=(tk, tv))
            assert st == kvx.KVX_OK
            assert torch.equal(tk, ref_k) and torch.equal(tv, ref_v), name
    finally:
        kvx.kvx_destroy(ctx)


# -------------------------------------------------------- cross-head (NEXT-1) -----

@pytest.mark.parametrize("over", [
    dict(Ls=3, Lt=4, H=2, B=1, T=300, k=2),                # ragged tail, odd tile count
    dict(Ls=5, Lt=3, H=4, B=2, T=129, k=3, theta_t=5e5),   # B > 1, different thetas, 1-row tail
    dict(Ls=4, Lt=2, H=2, B=1, T=1, k=1),                  # one token
    dict(Ls=6, Lt=3, H=8, B=1, T=256, k=4),                # eight heads, two full tiles
    dict(Ls=9, Lt=2, H=2, B=1, T=200, k=8, scores="uniform"),   # k = 8: 16 K steps, random selection
])
def test_cross_head_tc_small(over):
    """Cross-head tensor-core path (key strip, pair GEMM, epilogue) against the float64
    oracle on every output element, three launches each."""
    w = syn.workload("qwen3_14b_32b_t32768_k4_xhead", **over)
    ctx, sel, W, b = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b)
        for rep in range(3):
            tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
            assert st == kvx.KVX_OK
            ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
            assert ok, "launch %d: %d elements out of tolerance (worst %.3g x bound)" % (rep, nbad, ratio)
    finally:
        kvx.kvx_destroy(ctx)


@pytest.mark.parametrize("kname", ["simt", "tc"])
def test_cross_head_paged_small_full(kname):
    """The paper's cross-head mapper writing into a paged cache (16-token blocks, unaligned
    starts, a block table per sequence): every slot of two turns against the oracle, untouched
    slots keep their sentinel; the tensor-core kernel is also launched repeatedly."""
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", Ls=4, Lt=3, H=2, B=3, T=150, k=2,
                     len_range=(3, 70), head_mix="cross_head")
    ctx, sel, W, b = make_ctx(w, kernel=KERNELS[kname])
    try:
        L0 = syn.initial_lengths(w)
        rows = np.array([(bb, t) for bb in range(w.B) for t in range(w.T)], dtype=np.int64)
        for turn in (0, 1, 0, 1):
            _check_paged(w, ctx, sel, W, b, turn, L0, rows)
    finally:
        kvx.kvx_destroy(ctx)


def test_cross_head_paged_full_size_sampled():
    """Cross-head mapper (k = 4, every KV head of the selected layers) into the paged
    Qwen3-32B -> 14B turn (16 x 2048 new tokens at their absolute positions) on the tensor
    cores: sampled rows against the oracle, every slot checked."""
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", head_mix="cross_head")
    ctx, sel, W, b = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05)
    try:
        _check_paged(w, ctx, sel, W, b, 3, syn.initial_lengths(w), sample_rows(w, 24, seed=3))
    finally:
        kvx.kvx_destroy(ctx)
        torch.cuda.empty_cache()


def test_cross_head_full_size_sampled():
    """The cross-head bench workload (Qwen3-14B -> 32B shapes, k = 4, 32768 tokens): sampled
    rows against the oracle, every row written."""
    w = syn.workload("qwen3_14b_32b_t32768_k4_xhead")
    ctx, sel, W, b = make_ctx(w)
    dev = torch.device("cuda:0")
    try:
        sk = syn.source_cache(w, 0, device=dev)
        sv = syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        del sk, sv
        assert not torch.isnan(tk).any() and not torch.isnan(tv).any(), "unwritten rows"
        rows = sample_rows(w, 6)
        rk, rv, ak, av = oracle_rows(w, rows, pos, sel, W, b)
        gk = to_f64(tk[:, rows[:, 0], :, rows[:, 1]].permute(1, 2, 0, 3))
        gv = to_f64(tv[:, rows[:, 0], :, rows[:, 1]].permute(1, 2, 0, 3))
        ok, ratio, rms, nbad = check(w, [gk, gv], [rk, rv], [ak, av])
        assert ok, "%d sampled elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
    finally:
        kvx.kvx_destroy(ctx)
        torch.cuda.empty_cache()


# ------------------------------------------------------- Llama-3 frequency scaling -----

@pytest.mark.parametrize("kname", ["simt", "tc"])
def test_llama3_rope_scaling_small(kname):
    """Llama 3.1 shapes (theta 5e5) with the llama3 frequency scaling on both models, at
    positions past 10^5 so that the rescaled low frequencies turn: every output against the
    oracle (whose inverse frequencies follow the scaling's definition), and the result
    differs from the unscaled map."""
    over = dict(Ls=6, Lt=5, H=2, B=2, T=300, k=3, theta_s=5e5, theta_t=5e5)
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", rope_scaling=(8.0, 1.0, 4.0, 8192.0), **over)
    _kernel_or_skip(w, KERNELS[kname])
    ctx, sel, W, b = make_ctx(w, kernel=KERNELS[kname])
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w) + np.array([[123457], [250001]], dtype=np.int32)
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
        assert ok, "%d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
        plain = syn.workload("qwen3_14b_32b_b8x1024_k4", **over)
        pk, _, _, _ = oracle_full(plain, sk, sv, pos, sel, W, b)
        assert np.max(np.abs(pk - rk)) > 0.1 * rms          # the scaling does change the keys
    finally:
        kvx.kvx_destroy(ctx)


# ------------------------------------------------------------ host-buffer pipeline -----

@pytest.mark.parametrize("name,over,kernel,chunk", [
    ("qwen3_14b_32b_b8x1024_k4", dict(Ls=6, Lt=5, H=2, B=2, T=1000, k=3), "tc", 300),     # ragged chunks
    ("qwen3_14b_32b_b8x1024_k4", dict(Ls=6, Lt=5, H=2, B=2, T=1000, k=3), "simt", 256),
    ("qwen3_14b_32b_t32768_k4_xhead", dict(Ls=4, Lt=3, H=2, B=1, T=700, k=2), "tc", 128),
    ("qwen3_14b_32b_b8x1024_k4", dict(Ls=3, Lt=2, H=1, B=1, T=50, k=1), "tc", 4096),      # one short chunk
])
def test_map_host_equals_device_map(name, over, kernel, chunk):
    """kvx_map_host (pinned host caches, chunked, copies overlapped with the map) writes the
    same bytes into the host targets as kvx_map on device copies, over two calls through
    one pipe."""
    w = syn.workload(name, **over)
    ctx, sel, W, b = make_ctx(w, kernel=KERNELS[kernel])
    pipe = None
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w) + 17
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        hk, hv = sk.cpu().pin_memory(), sv.cpu().pin_memory()
        hpos = torch.from_numpy(np.ascontiguousarray(pos, dtype=np.int32)).pin_memory()
        pipe = kvx.kvx_host_pipe_create(ctx, w.B, chunk)
        s = torch.cuda.current_stream()
        untouched = torch.full(tk.shape, 3.0, dtype=tk.dtype).pin_memory()
        kvx.kvx_map_host(pipe, kvx.src_from_tensors(hk, hv), 0, hpos.data_ptr(),
                         kvx.tgt_from_tensors(untouched, untouched), s.cuda_stream)   # T = 0: no-op
        s.synchronize()
        assert torch.all(untouched == 3.0)
        for rep in range(2):
            ok_ = torch.full(tk.shape, float("nan"), dtype=tk.dtype).pin_memory()
            ov_ = torch.full(tv.shape, float("nan"), dtype=tv.dtype).pin_memory()
            kvx.kvx_map_host(pipe, kvx.src_from_tensors(hk, hv), w.T, hpos.data_ptr(),
                             kvx.tgt_from_tensors(ok_, ov_), s.cuda_stream)
            s.synchronize()
            assert kvx.kvx_get_status(ctx, s.cuda_stream) == kvx.KVX_OK
            assert torch.equal(ok_.view(torch.int16), tk.cpu().view(torch.int16)), rep
            assert torch.equal(ov_.view(torch.int16), tv.cpu().view(torch.int16)), rep
    finally:
        if pipe:
            kvx.kvx_host_pipe_destroy(pipe)
        kvx.kvx_destroy(ctx)


# ------------------------------------------------ fp32 weights on the tensor cores -----

def test_cross_head_tc_fp32_weights_hi_lo():
    """Cross-head tensor-core kernel with fp32 W (the paper keeps W in fp32): W^T is split
    into bf16 hi + lo and the K loop runs twice over the source tiles, so the result follows
    the fp32 weights.  Every output within the usual bound of the oracle given the fp32 W;
    at least 90 % of them equal to the correctly rounded fp32-W result (the rest sit within
    accumulation error of a rounding midpoint), where W rounded to bf16 gets visibly fewer."""
    w = syn.workload("qwen3_14b_32b_t32768_k4_xhead", Ls=4, Lt=3, H=2, B=1, T=300, k=2)
    Wb, b = syn.weights(w)
    g = torch.Generator().manual_seed(5)
    # fp32 weights off the bf16 grid, with a same-sign residual so that it shows in sums
    W32 = (Wb.float() * (1.0 + 2.0 ** -9 * (0.5 + 0.5 * torch.rand(Wb.shape, generator=g)))).contiguous()
    ctx, sel, _, _ = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05, W=W32, b=b)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W32, b)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
        assert ok, "%d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
        from oracle import bf16 as obf16
        gv = to_f64(tv)
        exact = np.mean(gv == obf16.round_to_bf16_value(rv))
        hk_, hv_ = oracle_full(w, sk, sv, pos, sel, Wb, b)[:2]     # W rounded to bf16
        hi_only = np.mean(obf16.round_to_bf16_value(hv_) == obf16.round_to_bf16_value(rv))
        assert exact >= 0.9 and exact > hi_only + 0.05, (exact, hi_only)
    finally:
        kvx.kvx_destroy(ctx)


@pytest.mark.parametrize("over", [
    dict(Ls=6, Lt=5, H=2, B=2, T=300, k=3),                 # ragged tail, B > 1
    dict(Ls=8, Lt=9, H=2, B=1, T=256, k=4, scores="uniform"),  # k = 4, reloads
    dict(Ls=9, Lt=3, H=4, B=1, T=200, k=6),                 # k = 6: cross-head kernel, per-head steps, W_lo pass
])
def test_per_head_tc_fp32_weights_hi_lo(over):
    """Per-head tensor-core kernel with fp32 W: each use takes a hi and a lo W stage over
    the same source tile, so the result follows the fp32 weights.  Every output within the
    usual bound of the oracle given the fp32 W; at least 90 % of the values equal to the
    correctly rounded fp32-W result, where W rounded to bf16 gets visibly fewer."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", **over)
    _kernel_or_skip(w, kvx.KVX_KERNEL_TCGEN05)
    Wb, b = syn.weights(w)
    g = torch.Generator().manual_seed(6)
    W32 = (Wb.float() * (1.0 + 2.0 ** -9 * (0.5 + 0.5 * torch.rand(Wb.shape, generator=g)))).contiguous()
    ctx, sel, _, _ = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05, W=W32, b=b)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W32, b)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
        assert ok, "%d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
        from oracle import bf16 as obf16
        exact = np.mean(to_f64(tv) == obf16.round_to_bf16_value(rv))
        hv_ = oracle_full(w, sk, sv, pos, sel, Wb, b)[1]     # W rounded to bf16
        hi_only = np.mean(obf16.round_to_bf16_value(hv_) == obf16.round_to_bf16_value(rv))
        assert exact >= 0.9 and exact > hi_only + 0.05, (exact, hi_only)
    finally:
        kvx.kvx_destroy(ctx)


# ------------------------------------------------------------------ CUDA graphs -----

@pytest.mark.parametrize("kname,name", [("simt", "qwen3_14b_32b_b8x1024_k4"), ("tc", "qwen3_14b_32b_b8x1024_k4"),
                                        ("tc", "qwen3_14b_32b_t32768_k4_xhead")])
def test_map_captured_in_a_cuda_graph(kname, name):
    """kvx_map captured into a CUDA graph (the cross-head kernel after one eager call has
    allocated its workspace): replays map whatever the captured buffers hold at replay
    time, bit for bit as eager calls on the same inputs, and the status stays OK."""
    w = syn.workload(name, Ls=5, Lt=3, H=2, B=2, T=300, k=2)
    ctx, sel, W, b = make_ctx(w, kernel=KERNELS[kname])
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = torch.from_numpy(syn.positions(w)).to(dev)
        tk = torch.full((w.Lt, w.B, w.H, w.T, w.d), float("nan"), dtype=torch.bfloat16, device=dev)
        tv = torch.full_like(tk, float("nan"))
        src, tgt = kvx.src_from_tensors(sk, sv), kvx.tgt_from_tensors(tk, tv)
        s = torch.cuda.Stream()
        with torch.cuda.stream(s):
            kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, s.cuda_stream)   # eager reference
        s.synchronize()
        ek, ev = tk.clone(), tv.clone()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, s.cuda_stream)
        for rep in range(2):
            tk.fill_(float("nan"))
            tv.fill_(float("nan"))
            g.replay()
            torch.cuda.synchronize()
            assert torch.equal(tk, ek) and torch.equal(tv, ev), "replay %d differs from the eager map" % rep
        # new inputs written into the captured buffers: the replay maps them
        sk.copy_(sk.flip(3))
        sv.copy_(sv.flip(3))
        pos.copy_(pos + 1000)
        g.replay()
        torch.cuda.synchronize()
        gk, gv = tk.clone(), tv.clone()
        with torch.cuda.stream(s):
            kvx.kvx_map(ctx, src, w.B, w.T, pos.data_ptr(), tgt, s.cuda_stream)
        s.synchronize()
        assert torch.equal(gk, tk) and torch.equal(gv, tv)
        assert not torch.equal(gk, ek)
        assert kvx.kvx_get_status(ctx, s.cuda_stream) == kvx.KVX_OK
        del g
    finally:
        kvx.kvx_destroy(ctx)


# ---------------------------------------------------------------- HF RoPE numerics -----

@pytest.mark.parametrize("kname", ["simt", "tc"])
def test_hf_rope_numerics(kname):
    """KVX_ROPE_HF (the rounding of the Hugging Face bf16 forward: fp32 angle, bf16 cos/sin,
    each product and sum rounded) on the SIMT and the per-head tensor-core kernels against
    the oracle in the same numerics, at positions past 2 * 10^4 where the fp32 angle is
    coarse: every output within the bound, at least 90 % of the keys bit-equal to the
    oracle's (the rest follow a rounding of the fp32-accumulated contraction or of cos / sin
    near a bf16 midpoint), far more than agree with the exact-RoPE oracle."""
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=5, Lt=4, H=2, B=2, T=200, k=2, theta_t=5e5)
    W, b = syn.weights(w)
    scores = syn.selection_scores(w)
    cfg, keep = kvx.config_from_tensors(
        src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k, theta_s=w.theta_s,
        theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b, scores=scores, rope_numerics=kvx.KVX_ROPE_HF)
    ctx = kvx.kvx_create(cfg, 0)
    try:
        kvx.kvx_set_kernel(ctx, KERNELS[kname])
        sel = kvx.kvx_get_selection(ctx, w.Lt, w.k)
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w) + np.array([[20011], [31007]], dtype=np.int32)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        sk64, sv64 = to_f64(sk), to_f64(sv)
        rk, rv = omap.map_cache(sk64, sv64, pos, sel, to_f64(W), to_f64(b), w.theta_s, w.theta_t,
                                mode="bf16fwd", rope_numerics="hf")
        ek, ev = omap.map_cache(sk64, sv64, pos, sel, to_f64(W), to_f64(b), w.theta_s, w.theta_t,
                                mode="bf16fwd")
        gk, gv = to_f64(tk), to_f64(tv)
        ok, ratio, rms, nbad = check(w, [gv], [rv])
        assert ok, "values: %d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
        # keys: a rounding taken on the other side of a bf16 midpoint (the mapped key before
        # the rotation, or cos / sin) moves an output by a few bf16 steps of its pair's terms,
        # so the bound scales with the pair magnitude |a| + |b| (4 steps: 2^-6 of it)
        mag = np.concatenate([np.abs(rk[..., :64]) + np.abs(rk[..., 64:])] * 2, axis=-1)
        err = np.abs(gk - rk)
        assert np.all(err <= 2.0 ** -6 * mag + 1e-3 * rms), np.max(err / (2.0 ** -6 * mag + 1e-3 * rms))
        from oracle import bf16 as obf16
        same_hf = np.mean(gk == rk)
        same_exact = np.mean(gk == obf16.round_to_bf16_value(ek))
        assert same_hf >= 0.9 and same_hf > same_exact + 0.1, (same_hf, same_exact)
    finally:
        kvx.kvx_destroy(ctx)


def test_hf_rope_numerics_cross_head_tc():
    """KVX_ROPE_HF on the cross-head tensor-core kernel (HF strip in the key-strip kernel, HF
    rotation in the epilogue): every output within the bound of the HF oracle and at least
    90 % of the keys bit-equal to it, far more than agree with the exact-RoPE oracle."""
    w = syn.workload("qwen3_14b_32b_t32768_k4_xhead", Ls=4, Lt=3, H=2, B=1, T=300, k=2, theta_t=5e5)
    W, b = syn.weights(w)
    cfg, keep = kvx.config_from_tensors(
        src_layers=w.Ls, tgt_layers=w.Lt, n_kv_heads=w.H, head_dim=w.d, k=w.k, theta_s=w.theta_s,
        theta_t=w.theta_t, cache_dtype=w.cache_dtype, W=W, b=b, scores=syn.selection_scores(w),
        head_mix=kvx.KVX_CROSS_HEAD, rope_numerics=kvx.KVX_ROPE_HF)
    ctx = kvx.kvx_create(cfg, 0)
    try:
        kvx.kvx_set_kernel(ctx, kvx.KVX_KERNEL_TCGEN05)
        sel = kvx.kvx_get_selection(ctx, w.Lt, w.k)
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w) + 20011
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        sk64, sv64 = to_f64(sk), to_f64(sv)
        common = dict(mode="bf16fwd", head_mix="cross_head")
        rk, rv = omap.map_cache(sk64, sv64, pos, sel, to_f64(W), to_f64(b), w.theta_s, w.theta_t,
                                rope_numerics="hf", **common)
        ek, _ = omap.map_cache(sk64, sv64, pos, sel, to_f64(W), to_f64(b), w.theta_s, w.theta_t, **common)
        gk, gv = to_f64(tk), to_f64(tv)
        ok, ratio, rms, nbad = check(w, [gv], [rv])
        assert ok, "values: %d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
        mag = np.concatenate([np.abs(rk[..., :64]) + np.abs(rk[..., 64:])] * 2, axis=-1)
        assert np.all(np.abs(gk - rk) <= 2.0 ** -6 * mag + 1e-3 * rms)
        from oracle import bf16 as obf16
        same_hf, same_exact = np.mean(gk == rk), np.mean(gk == obf16.round_to_bf16_value(ek))
        assert same_hf >= 0.9 and same_hf > same_exact + 0.1, (same_hf, same_exact)
    finally:
        kvx.kvx_destroy(ctx)


# ------------------------------------------------------------ bounded waits -----

def test_bounded_wait_runs_out_and_the_context_recovers():
    """The tensor-core kernel's abort path, on a healthy GPU: with the test switch its first
    CTA never loads one bias row, so the epilogue's wait for it runs out after the shortened
    50 ms bound.  The launch must end by itself (well within a second), the status word
    must read KVX_ERR_TIMEOUT, and the next launch on the same context (switch off) must map
    every element within the oracle's tolerance."""
    import time
    w = syn.workload("qwen3_14b_32b_b8x1024_k4", Ls=3, Lt=4, H=1, B=1, T=256, k=2)
    ctx, sel, W, b = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        pos = syn.positions(w)
        torch.cuda.synchronize()
        kvx.kvx_set_test_wait(ctx, 50_000_000, skip_bias_row=1)
        t0 = time.perf_counter()
        tk, tv, status = run_contiguous(ctx, w, sk, sv, pos)
        dt = time.perf_counter() - t0
        assert status == kvx.KVX_ERR_TIMEOUT, kvx.kvx_status_string(status)
        assert dt < 1.0, "the aborted launch took %.3f s" % dt
        kvx.kvx_set_test_wait(ctx, 0, -1)
        tk, tv, status = run_contiguous(ctx, w, sk, sv, pos)
        assert status == kvx.KVX_OK
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b)
        ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
        assert ok, "after the abort: %d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
    finally:
        kvx.kvx_destroy(ctx)


# ------------------------------------------------- multi-turn persistent pool -----

def _persistent_turns(w, kname, rows_of_turn, check_sentinel_turns):
    """Map all w.turns turns into one pool whose block table covers every sequence's final
    length (Sec. 4.5: only each turn's new tokens are mapped, at their absolute positions).
    After each turn: the checked rows of every turn so far equal the oracle (a later turn
    must not disturb them), and, on the turns listed, every slot outside the positions
    mapped so far keeps its sentinel while every mapped slot is fully written."""
    ctx, sel, W, b = make_ctx(w, kernel=KERNELS[kname])
    dev = torch.device("cuda:0")
    try:
        L0 = syn.initial_lengths(w)
        table, n_blocks = syn.persistent_block_table(w, L0)
        tbl = torch.from_numpy(table).to(dev)
        pool_k = torch.empty((w.Lt, n_blocks, w.H, w.block_size, w.d), dtype=torch.bfloat16, device=dev)
        pool_v = torch.empty_like(pool_k)
        pool_k.view(torch.int16).fill_(0x7FBF)
        pool_v.view(torch.int16).fill_(0x7FBF)
        tgt = kvx.tgt_paged_from_tensors(pool_k, pool_v, tbl, w.block_size)
        written = torch.zeros((n_blocks, w.block_size), dtype=torch.bool)
        s = torch.cuda.current_stream().cuda_stream
        refs = []
        for turn in range(w.turns):
            pos = syn.positions(w, turn, L0)
            sk = syn.source_cache(w, 0, device=dev, turn=turn)
            sv = syn.source_cache(w, 1, device=dev, turn=turn)
            posd = torch.from_numpy(pos).to(dev)
            kvx.kvx_map(ctx, kvx.src_from_tensors(sk, sv), w.B, w.T, posd.data_ptr(), tgt, s)
            assert kvx.kvx_get_status(ctx, s) == kvx.KVX_OK, "turn %d" % turn
            del sk, sv
            for bb in range(w.B):
                written[torch.from_numpy(table[bb, pos[bb] // w.block_size].astype(np.int64)),
                        torch.from_numpy((pos[bb] % w.block_size).astype(np.int64))] = True
            rows = rows_of_turn(turn)
            rk, rv, ak, av = oracle_rows(w, rows, pos, sel, W, b, turn=turn)
            p = pos[rows[:, 0], rows[:, 1]]
            refs.append((rows, table[rows[:, 0], p // w.block_size].astype(np.int64),
                         (p % w.block_size).astype(np.int64), rk, rv, ak, av))
            for j, (rows_j, blk, slot, rk, rv, ak, av) in enumerate(refs):
                gk = to_f64(pool_k[:, blk, :, slot].permute(1, 2, 0, 3))
                gv = to_f64(pool_v[:, blk, :, slot].permute(1, 2, 0, 3))
                ok, ratio, rms, nbad = check(w, [gk, gv], [rk, rv], [ak, av])
                assert ok, "after turn %d, rows of turn %d: %d out of tolerance (worst %.3g)" % (turn, j, nbad, ratio)
            if turn in check_sentinel_turns:
                wd = written.to(dev)
                for pool in (pool_k, pool_v):
                    for l in range(w.Lt):          # one layer at a time bounds the temporaries
                        sent = pool[l].view(torch.int16) == 0x7FBF            # [nb][H][bs][d]
                        assert torch.equal(sent.all(dim=-1).all(dim=1), ~wd), \
                            "turn %d layer %d: a slot outside the mapped tokens was touched" % (turn, l)
                        assert torch.equal((~sent).all(dim=-1).all(dim=1), wd), \
                            "turn %d layer %d: a mapped slot was not fully written" % (turn, l)
                        del sent
    finally:
        kvx.kvx_destroy(ctx)
        torch.cuda.empty_cache()


@pytest.mark.parametrize("kname", ["simt", "tc"])
def test_paged_persistent_pool_eight_turns_small(kname):
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", Ls=5, Lt=3, H=2, B=3, T=37, k=2,
                     len_range=(3, 70))
    if kname == "tc":
        _kernel_or_skip(w, KERNELS[kname])
    every_row = np.array([(bb, t) for bb in range(w.B) for t in range(w.T)], dtype=np.int64)
    _persistent_turns(w, kname, lambda turn: every_row, check_sentinel_turns=range(w.turns))


def test_paged_persistent_pool_eight_turns_full_size_sampled():
    """The Qwen3-32B -> 14B paged workload as specified: 16 sequences, initial lengths in
    [2048, 16384], eight turns of 2048 new tokens into one pool sized for the final lengths
    (about 67 GB of bf16 target cache); 24 sampled rows per turn, all earlier turns'
    sampled rows re-checked after each turn, every slot checked after the first and the
    last turn."""
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4")
    _persistent_turns(w, "tc", lambda turn: sample_rows(w, 24, seed=100 + turn),
                      check_sentinel_turns=(0, w.turns - 1))


# ------------------------------------------------- tensor cores at large positions -----

@pytest.mark.parametrize("name,style", [("qwen3_14b_32b_b8x1024_k4", "half"), ("qwen3_14b_32b_b8x1024_k4", "interleaved"),
                                        ("qwen3_14b_32b_t32768_k4_xhead", "half")])
def test_tensor_cores_up_to_max_position(name, style):
    """The tensor-core kernels at positions spread over [0, 2^24) including 2^24 - 1 (the
    largest accepted) and powers of two with their neighbours: every output element within
    the bf16 bound of the oracle (with the strip's rounding slack), values and keys."""
    w = syn.workload(name, Ls=5, Lt=3, H=2, B=2, T=300, k=2, theta_t=5e5, rope_style=style)
    rng = np.random.default_rng(7)
    special = [0, 1, (1 << 24) - 1, (1 << 24) - 2] + [(1 << e) + o for e in range(10, 24) for o in (-1, 0, 1)]
    flat = np.array(special + list(rng.integers(0, 1 << 24, size=w.B * w.T - len(special))), dtype=np.int32)
    pos = flat.reshape(w.B, w.T)
    ctx, sel, W, b = make_ctx(w, kernel=kvx.KVX_KERNEL_TCGEN05)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        rk, rv, ak, av = oracle_full(w, sk, sv, pos, sel, W, b)
        ok, ratio, rms, nbad = check(w, [to_f64(tk), to_f64(tv)], [rk, rv], [ak, av])
        assert ok, "%d elements out of tolerance (worst %.3g x bound)" % (nbad, ratio)
    finally:
        kvx.kvx_destroy(ctx)


# ------------------------------------------------------------ strip error bound -----

def test_strip_error_within_delta_up_to_max_position():
    """Pins STRIP_DELTA, the per-rotation error the rounding slack of the bf16 tests assumes:
    a stored pair (a, b) rotated by the kernels' angle arithmetic (float-float angle,
    Cody-Waite reduction, sincosf) is within delta (|a| + |b|) of the exact rotation.  With
    fp32 caches, k = 1, W = I, b = 0 and theta_s != theta_t the map is two such rotations (strip
    by theta_s, re-rotation by theta_t); the second acts on a pair of size at most
    sqrt(2) (|a| + |b|) and rotations preserve the first one's error, so every key output is
    within 2 sqrt(2) delta (|a| + |b|) of the exact oracle (plus one fp32 rounding).  Positions
    cover 0, powers of two and their neighbours, random values and 2^24 - 1 (the largest
    accepted); values must come back bit for bit."""
    from harness import STRIP_DELTA
    w = syn.workload("tiny_fp32", Ls=1, Lt=1, H=1, d=128, k=1, B=1, T=1024, theta_s=1e6, theta_t=5e5)
    rng = np.random.default_rng(24)
    special = [0, 1, 2, 3, (1 << 24) - 1, (1 << 24) - 2] + [(1 << e) + o for e in range(2, 24) for o in (-1, 0, 1)]
    pos = np.array(special + list(rng.integers(0, 1 << 24, size=w.T - len(special))), dtype=np.int32)[None, :]
    W = torch.zeros((1, 2, 1, 128, 128), dtype=torch.float32)
    W[0, :, 0] = torch.eye(128)
    b = torch.zeros((1, 2, 1, 128), dtype=torch.float32)
    ctx, sel, _, _ = make_ctx(w, selection=np.zeros((1, 1), dtype=np.int32), W=W, b=b)
    try:
        dev = torch.device("cuda:0")
        sk, sv = syn.source_cache(w, 0, device=dev), syn.source_cache(w, 1, device=dev)
        tk, tv, st = run_contiguous(ctx, w, sk, sv, pos)
        assert st == kvx.KVX_OK
        assert torch.equal(tv, sv), "values must pass through W = I unchanged"
        x = to_f64(sk)[0, 0, 0]                                  # [T][128] stored keys
        ref = omap.map_tokens(x[None, None], to_f64(sv)[0, 0, 0][None, None], pos[0], sel, W.double().numpy(),
                              b.double().numpy(), w.theta_s, w.theta_t, mode="exact")[0][0, 0]   # [T][128]
        got = to_f64(tk)[0, 0, 0]
        mag = np.abs(x[:, :64]) + np.abs(x[:, 64:])
        mag = np.concatenate([mag, mag], axis=1)                 # |a| + |b| of each output's pair
        bound = 2.0 * np.sqrt(2.0) * STRIP_DELTA * mag + 2.0 ** -23 * np.abs(ref)
        err = np.abs(got - ref)
        ratio = err / bound
        assert np.all(err <= bound), "worst %.3g x bound at position %d" % (
            ratio.max(), pos[0, np.unravel_index(np.argmax(ratio), ratio.shape)[0]])
        assert np.array_equal(got[0], x[0]), "position 0 must come back unrotated and exact"
    finally:
        kvx.kvx_destroy(ctx)
