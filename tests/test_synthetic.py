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
