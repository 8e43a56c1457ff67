"""The shared input generator: deterministic, row-addressable, CPU-only checks."""
import numpy as np
import torch

from paper_2608_03893_gb300 import synthetic as syn


def test_splitmix64_known_values():
    # SplitMix64 seeded with 0: the first outputs of the published generator
    # (state advanced by the golden gamma before each output).
    g = 0x9E3779B97F4A7C15
    outs = [syn.splitmix64_py((g * (n + 1)) & ((1 << 64) - 1)) for n in range(3)]
    assert outs == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_torch_generator_matches_pure_python():
    key = syn.stream_key(5, 3)
    idx = torch.tensor([0, 1, 2, 1000, 123456789, (1 << 40) + 7], dtype=torch.int64)
    got = syn.irwin_hall12(key, idx).tolist()
    for i, g in zip(idx.tolist(), got):
        assert g == syn.irwin_hall12_py(key, i)


def test_torch_generator_matches_pure_python_over_many_indices():
    # every bit of the 64-bit words gets both values over a few hundred indices and keys
    for seed, stream in ((5, 3), (0, 1), (7, 104)):
        key = syn.stream_key(seed, stream)
        got = syn.irwin_hall12(key, torch.arange(256)).tolist()
        assert got == [syn.irwin_hall12_py(key, i) for i in range(256)], (seed, stream)


def test_irwin_hall_moments():
    z = syn.irwin_hall12(syn.stream_key(1, 1), torch.arange(1 << 20)).double()
    assert abs(z.mean().item()) < 5e-3
    assert abs(z.var().item() - 1.0) < 5e-3
    assert z.abs().max().item() < 6.0


def test_source_rows_match_full_cache():
    w = syn.workload("tiny_fp32")
    for kv in (0, 1):
        full = syn.source_cache(w, kv)
        rows = np.array([[0, 0], [0, 17], [0, 255]])
        part = syn.source_rows(w, kv, rows)
        for n, (b, t) in enumerate(rows):
            assert torch.equal(part[:, :, n], full[:, b, :, t])


def test_bf16_rows_match_full_cache():
    w = syn.workload("tiny_fp32", cache_dtype="bf16", B=2, T=40, Ls=3)
    full = syn.source_cache(w, 0)
    assert full.dtype == torch.bfloat16
    rows = np.array([[1, 39], [0, 3]])
    part = syn.source_rows(w, 0, rows)
    for n, (b, t) in enumerate(rows):
        assert torch.equal(part[:, :, n], full[:, b, :, t])


def test_weights_scores_positions_shapes():
    w = syn.workload("tiny_fp32")
    W, b = syn.weights(w)
    assert W.shape == (6, 2, 2, 128, 64) and b.shape == (6, 2, 2, 64)
    assert abs(W.double().std().item() - (1 / 128) ** 0.5) < 0.01
    assert abs(b.double().std().item() - 0.1) < 0.02
    S = syn.selection_scores(w)
    assert S.shape == (6, 4)
    pos = syn.positions(w)
    assert pos.shape == (1, 256) and pos[0, 0] == 0 and pos[0, -1] == 255


def test_paged_block_table_is_a_permutation():
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4")
    L0 = syn.initial_lengths(w)
    assert L0.min() >= 2048 and L0.max() <= 16384
    for turn in (0, 7):
        pos = syn.positions(w, turn, L0)
        table, n_blocks = syn.block_table(w, pos, turn)
        used = table[table >= 0]
        assert sorted(used.tolist()) == list(range(n_blocks))
        for b in range(w.B):
            assert np.all(table[b, pos[b] // 16] >= 0)


def test_persistent_block_table_is_a_permutation_over_final_lengths():
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", B=5, T=37, len_range=(3, 70))
    L0 = syn.initial_lengths(w)
    table, n_blocks = syn.persistent_block_table(w, L0)
    final = L0 + w.turns * w.T
    nb = (final + w.block_size - 1) // w.block_size
    assert n_blocks == nb.sum() and table.shape == (w.B, nb.max())
    used = np.concatenate([table[b, :nb[b]] for b in range(w.B)])
    assert np.array_equal(np.sort(used), np.arange(n_blocks))
    for b in range(w.B):
        assert np.all(table[b, nb[b]:] == -1)
    # every position any turn maps has a block
    for turn in range(w.turns):
        pos = syn.positions(w, turn, L0)
        assert np.all(table[np.arange(w.B)[:, None], pos // w.block_size] >= 0)


def test_workload_defaults_positions_and_streams():
    for name, w in syn.WORKLOADS.items():
        pos = syn.positions(w) if not w.paged else None
        if not w.paged:
            assert w.turns == 1 and w.len_range == (0, 0), name
            assert np.array_equal(pos, np.tile(np.arange(w.T, dtype=np.int32), (w.B, 1))), name
    assert [n for n, w in syn.WORKLOADS.items() if w.paged] == ["qwen3_32b_14b_paged_b16_turn2048_k4"]
    assert syn.WORKLOADS["qwen3_32b_14b_paged_b16_turn2048_k4"].turns == 8
    # K and V, every turn and the fit's target cache draw from different streams
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", Ls=2, Lt=3, H=2, B=2, T=8)
    rows = np.array([[0, 0], [1, 5]])
    draws = [syn.source_rows(w, kv, rows, turn=t) for t in (None, 0, 1) for kv in (0, 1)]
    for i in range(len(draws)):
        for j in range(i):
            assert not torch.equal(draws[i], draws[j]), (i, j)
    # stream ids: the fixed ones (scales, caches, W, b, scores, lengths, blocks) and one per
    # (turn, K|V) of the paged workload, all different
    ids = [syn.STREAM_SCALE_K, syn.STREAM_SCALE_V, syn.STREAM_CACHE_K, syn.STREAM_CACHE_V, syn.STREAM_W,
           syn.STREAM_B, syn.STREAM_SCORES, syn.STREAM_LENGTHS, syn.STREAM_BLOCKS]
    ids += [syn._cache_stream(kv, t) for t in range(64) for kv in (0, 1)]
    assert len(set(ids)) == len(ids)
    assert syn._cache_stream(0, None) == syn.STREAM_CACHE_K and syn._cache_stream(1, None) == syn.STREAM_CACHE_V
    tk = syn.target_cache(w, 0)
    assert tk.shape == (w.Lt, w.B, w.H, w.T, w.d)
    assert not torch.equal(tk[:w.Ls], syn.source_cache(w, 0))


def test_channel_scales_recipe():
    """lognormal(0, 0.5) per (source layer, head, channel), K and V apart, and exactly
    round(1 % of them) distinct entries multiplied by 8 (the outlier channels)."""
    w = syn.workload("qwen3_14b_32b_t32768_k4")
    sk, sv = syn.channel_scales(w)
    k0, v0 = syn.channel_scales(syn.workload("qwen3_14b_32b_t32768_k4", outlier_frac=0.0))
    assert sk.shape == (w.Ls, w.H, w.d) and not np.array_equal(sk, sv)
    for s, s0 in ((sk, k0), (sv, v0)):
        ratio = s.astype(np.float64) / s0
        assert np.all((np.abs(ratio - 1) < 1e-6) | (np.abs(ratio - 8) < 1e-5))
        assert np.sum(np.abs(ratio - 8) < 1e-5) == round(0.01 * s.size)
        lg = np.log(s0.astype(np.float64))
        assert abs(np.median(lg)) < 0.02 and abs(lg.std() - 0.5) < 0.01


def test_weight_and_score_recipes():
    w = syn.workload("qwen3_14b_32b_b8x1024_k4")
    W, b = syn.weights(w)
    assert abs(W.double().std().item() * w.F ** 0.5 - 1.0) < 0.01
    assert abs(b.double().std().item() - 0.1) < 0.005 and abs(b.double().mean().item()) < 0.005
    # proportional depth: exp(-(l'/(L_s-1) - l/(L_t-1))^2 / (2 0.05^2)) plus jitter in [0, 0.02)
    S = syn.selection_scores(w)
    lp = np.arange(w.Ls)[None, :] / (w.Ls - 1)
    l = np.arange(w.Lt)[:, None] / (w.Lt - 1)
    jitter = S - np.exp(-((lp - l) ** 2) / (2 * 0.05 ** 2))
    assert jitter.min() >= 0 and jitter.max() < 0.02 and jitter.max() > 0.015
    # the uniform recipe of the tiny workload: iid U(0, 1)
    S = syn.selection_scores(syn.workload("tiny_fp32"))
    assert S.min() >= 0 and S.max() < 1


def test_lengths_are_inclusive_and_block_tables_exact():
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", B=64, T=8, len_range=(5, 6))
    assert set(syn.initial_lengths(w).tolist()) == {5, 6}
    # a turn that starts past the first blocks: those stay -1, the touched ones are numbered
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", B=4, T=8, len_range=(40, 41))
    pos = syn.positions(w, 0, syn.initial_lengths(w))
    table, n_blocks = syn.block_table(w, pos)
    assert table.shape == (w.B, int(pos.max()) // 16 + 1)
    assert np.all(table[:, :2] == -1) and set(table[table < 0].tolist()) == {-1}
    # the persistent pool: exactly sum ceil(final / 16) blocks, every residue of final mod 16
    w = syn.workload("qwen3_32b_14b_paged_b16_turn2048_k4", B=16, T=16, turns=2)
    lengths = np.arange(16) + 3                      # final = 35 .. 50
    table, n_blocks = syn.persistent_block_table(w, lengths)
    final = lengths + 32
    assert n_blocks == int(sum(-(-f // 16) for f in final)) and table.shape == (16, 4)
