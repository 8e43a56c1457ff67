"""Seeded synthetic workloads for the KV mapper: inputs only, no arithmetic of the method.

The tests, the bench and the oracle checks all draw their inputs here, so the CUDA
path and the float64 oracle see byte-identical data.  Nothing in this module rotates,
selects, concatenates or contracts anything: it only draws numbers and lays them out.

Shapes follow the paper's model pairs (Appendix C, Table "Transfer pairs studied":
8 KV heads of dimension 128 for every pair; Qwen3 14B/32B have 40/64 layers, Llama-3.1
8B/70B have 32/80).  There are no model weights or calibration caches here, so the
value distributions are stand-ins:

* source cache values: Irwin-Hall(12) draws (the sum of twelve uniforms minus six, a
  classical bounded stand-in for N(0, 1)) times a per-(layer, head, channel) scale
  drawn from lognormal(0, 0.5); in the larger workloads 1% of (layer, head, channel)
  triples get an extra x8 outlier scale.  The stored key cache is drawn directly (not
  as rotated content vectors): the map strips whatever the cache holds.
* W ~ N(0, 1/F) and b ~ N(0, 0.01) (variance), F the feature width.
* selection scores: iid U(0, 1) (tiny workload) or "nearest to proportional depth"
  exp(-(l'/(L_s-1) - l/(L_t-1))^2 / (2 * 0.05^2)) + 0.02 U(0, 1).

The source caches can be many GB, so their values come from a counter-based generator
(the SplitMix64 output function of Steele, Lea and Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014) evaluated with torch integer ops: element
i of a tensor is a pure function of (seed, stream, i).  The same values come out on the
CPU and on the GPU, in full or for any chosen rows.  Small tensors (scales, W, b,
scores, lengths, block tables) come from numpy's PCG64 ``default_rng`` seeded by
(seed, stream).
"""
from dataclasses import dataclass, field, replace

import numpy as np
import torch

# ----------------------------------------------------------------------------------
# counter-based generator
_GOLDEN = 0x9E3779B97F4A7C15
_MUL1 = 0xBF58476D1CE4E5B9
_MUL2 = 0x94D049BB133111EB
_U64 = (1 << 64) - 1


def _as_i64(c):
    c &= _U64
    return c - (1 << 64) if c >= (1 << 63) else c


def splitmix64_py(x):
    """Reference SplitMix64 output function on a Python int (exact mod 2^64)."""
    z = x & _U64
    z = ((z ^ (z >> 30)) * _MUL1) & _U64
    z = ((z ^ (z >> 27)) * _MUL2) & _U64
    return z ^ (z >> 31)


def _mix64(z):
    """SplitMix64 output function on int64 tensors holding uint64 bit patterns."""
    z = (z ^ ((z >> 30) & ((1 << 34) - 1))) * _as_i64(_MUL1)
    z = (z ^ ((z >> 27) & ((1 << 37) - 1))) * _as_i64(_MUL2)
    return z ^ ((z >> 31) & ((1 << 33) - 1))


def stream_key(seed, stream):
    return _as_i64(splitmix64_py((seed << 32) ^ (stream * _GOLDEN)))


def irwin_hall12(key, idx):
    """Float32 draws for element indices ``idx`` (int64 tensor) of the stream ``key``.

    Two 64-bit words per element give twelve 10-bit uniforms u_j; the value is
    (sum_j u_j - 6138) / 1024, i.e. sum_j (u_j + 0.5)/1024 - 6: mean 0, variance
    1 - 2^-20, range (-6, 6).  Every step is integer or exact, so CPU and GPU agree bit
    for bit.
    """
    c = idx * 2
    h1 = _mix64(key + (c + 1) * _as_i64(_GOLDEN))
    h2 = _mix64(key + (c + 2) * _as_i64(_GOLDEN))
    s = torch.zeros_like(idx)
    for h in (h1, h2):
        for j in range(6):
            s += (h >> (10 * j)) & 1023
    return (s - 6138).to(torch.float32) * (1.0 / 1024.0)


def irwin_hall12_py(key, i):
    """Pure-Python restatement of ``irwin_hall12`` for one index (pins the torch ops)."""
    u = key & _U64
    s = 0
    for w in (1, 2):
        h = splitmix64_py(u + (2 * i + w) * _GOLDEN)
        s += sum((h >> (10 * j)) & 1023 for j in range(6))
    return (s - 6138) / 1024.0


# ----------------------------------------------------------------------------------
# workloads
STREAM_SCALE_K, STREAM_SCALE_V, STREAM_CACHE_K, STREAM_CACHE_V = 1, 2, 3, 4
STREAM_W, STREAM_B, STREAM_SCORES, STREAM_LENGTHS, STREAM_BLOCKS = 5, 6, 7, 8, 9
STREAM_TURN_BASE = 100   # per-turn caches of the paged workload: 100 + 2 * turn (+1 for V)


@dataclass(frozen=True)
class Workload:
    name: str
    Ls: int
    Lt: int
    H: int
    d: int
    k: int
    B: int
    T: int                      # tokens mapped per sequence (per turn when paged)
    theta_s: float
    theta_t: float
    cache_dtype: str            # "f32" | "bf16"
    weight_dtype: str           # "f32" | "bf16"
    scores: str                 # "uniform" | "depth"
    outlier_frac: float
    seed: int
    paged: bool = False
    turns: int = 1
    block_size: int = 16
    len_range: tuple = (0, 0)   # initial per-sequence lengths (paged), inclusive
    head_mix: str = "per_head"  # "per_head" (F = k d) | "cross_head" (F = k H d, the paper's)
    rope_scaling: tuple = ()    # Llama-3 frequency scaling of both models, or () for plain theta
    rope_style: str = "half"    # RoPE pairs: "half" (i, i + d/2) | "interleaved" (2i, 2i + 1)
    notes: str = field(default="", compare=False)

    @property
    def F(self):
        return self.k * self.d * (self.H if self.head_mix == "cross_head" else 1)

    @property
    def n_tokens(self):
        return self.B * self.T

    def torch_dtype(self, which="cache"):
        dt = self.cache_dtype if which == "cache" else self.weight_dtype
        return torch.float32 if dt == "f32" else torch.bfloat16


WORKLOADS = {
    "tiny_fp32": Workload("tiny_fp32", 4, 6, 2, 64, 2, 1, 256, 1e4, 1e4, "f32", "f32",
                          "uniform", 0.0, 0),
    "qwen3_14b_32b_b8x1024_k4": Workload("qwen3_14b_32b_b8x1024_k4", 40, 64, 8, 128, 4, 8, 1024,
                                         1e6, 1e6, "bf16", "bf16", "depth", 0.01, 1),
    "qwen3_14b_32b_t32768_k1": Workload("qwen3_14b_32b_t32768_k1", 40, 64, 8, 128, 1, 1, 32768,
                                        1e6, 1e6, "bf16", "bf16", "depth", 0.01, 2),
    "qwen3_14b_32b_t32768_k2": Workload("qwen3_14b_32b_t32768_k2", 40, 64, 8, 128, 2, 1, 32768,
                                        1e6, 1e6, "bf16", "bf16", "depth", 0.01, 2),
    "qwen3_14b_32b_t32768_k4": Workload("qwen3_14b_32b_t32768_k4", 40, 64, 8, 128, 4, 1, 32768,
                                        1e6, 1e6, "bf16", "bf16", "depth", 0.01, 2),
    "llama31_8b_70b_b4x8192_k3": Workload("llama31_8b_70b_b4x8192_k3", 32, 80, 8, 128, 3, 4, 8192,
                                          5e5, 5e5, "bf16", "bf16", "depth", 0.01, 3),
    "llama31_70b_8b_b4x8192_k3": Workload("llama31_70b_8b_b4x8192_k3", 80, 32, 8, 128, 3, 4, 8192,
                                          5e5, 5e5, "bf16", "bf16", "depth", 0.01, 3),
    "qwen3_32b_14b_paged_b16_turn2048_k4": Workload(
        "qwen3_32b_14b_paged_b16_turn2048_k4", 64, 40, 8, 128, 4, 16, 2048, 1e6, 1e6, "bf16",
        "bf16", "depth", 0.01, 4, paged=True, turns=8, block_size=16, len_range=(2048, 16384)),
    # the paper's mapper layout (every KV head of the selected layers feeds every target
    # head); k = 8 is the Qwen3 14B -> 32B pair of its latency table
    "qwen3_14b_32b_b8x1024_k4_xhead": Workload("qwen3_14b_32b_b8x1024_k4_xhead", 40, 64, 8, 128, 4, 8, 1024,
                                               1e6, 1e6, "bf16", "bf16", "depth", 0.01, 1, head_mix="cross_head"),
    "qwen3_14b_32b_t32768_k4_xhead": Workload("qwen3_14b_32b_t32768_k4_xhead", 40, 64, 8, 128, 4, 1, 32768,
                                              1e6, 1e6, "bf16", "bf16", "depth", 0.01, 2, head_mix="cross_head"),
    "qwen3_14b_32b_t32768_k8_xhead": Workload("qwen3_14b_32b_t32768_k8_xhead", 40, 64, 8, 128, 8, 1, 32768,
                                              1e6, 1e6, "bf16", "bf16", "depth", 0.01, 2, head_mix="cross_head"),
    # the MLP mapper's shapes (cross-head d_s = 4096, hidden 1024): 11 GFLOP per token, 45 TFLOP a step
    "qwen3_14b_32b_b1x4096_k4_xhead": Workload("qwen3_14b_32b_b1x4096_k4_xhead", 40, 64, 8, 128, 4, 1, 4096,
                                              1e6, 1e6, "bf16", "bf16", "depth", 0.01, 3, head_mix="cross_head"),
}

HEADLINE = "qwen3_14b_32b_t32768_k4"


def workload(name, **overrides):
    w = WORKLOADS[name]
    return replace(w, **overrides) if overrides else w


def _rng(w, stream):
    return np.random.default_rng([w.seed, stream])


def channel_scales(w):
    """(scale_k, scale_v): float32 [L_s][H][d] lognormal(0, 0.5), with outliers x8."""
    out = []
    for stream in (STREAM_SCALE_K, STREAM_SCALE_V):
        rng = _rng(w, stream)
        s = rng.lognormal(0.0, 0.5, size=(w.Ls, w.H, w.d))
        n_out = int(round(w.outlier_frac * s.size))
        if n_out:
            s.reshape(-1)[rng.choice(s.size, size=n_out, replace=False)] *= 8.0
        out.append(s.astype(np.float32))
    return out[0], out[1]


def _cache_stream(kv, turn):
    if turn is None:
        return STREAM_CACHE_K if kv == 0 else STREAM_CACHE_V
    return STREAM_TURN_BASE + 2 * turn + kv


def source_cache(w, kv, device="cpu", turn=None, out=None):
    """Full source cache [L_s][B][H][T][d] in the workload's cache dtype.

    ``kv`` 0 = keys, 1 = values.  ``turn`` selects the per-turn cache of the paged
    workload.  Generated one source layer at a time; ``out`` may be a preallocated
    tensor of the right shape (on any device) to fill.
    """
    key = stream_key(w.seed, _cache_stream(kv, turn))
    scale = torch.from_numpy(channel_scales(w)[kv]).to(device)
    shape = (w.Ls, w.B, w.H, w.T, w.d)
    if out is None:
        out = torch.empty(shape, dtype=w.torch_dtype(), device=device)
    per_layer = w.B * w.H * w.T * w.d
    for l in range(w.Ls):
        idx = torch.arange(l * per_layer, (l + 1) * per_layer, device=device, dtype=torch.int64)
        z = irwin_hall12(key, idx).view(w.B, w.H, w.T, w.d)
        val = z * scale[l].view(1, w.H, 1, w.d)
        out[l].copy_(val.to(out.dtype))
        del idx, z, val
    return out


def target_cache(w, kv, device="cpu"):
    """Calibration target cache [L_t][B][H][T][d] for a ridge fit: the source-cache recipe
    for L_t layers under seed w.seed + 1000 (independent of the source cache)."""
    return source_cache(replace(w, Ls=w.Lt, seed=w.seed + 1000, paged=False), kv, device=device)


def source_rows(w, kv, rows, turn=None):
    """Source values for chosen token rows, on the CPU, identical to ``source_cache``.

    ``rows``: int array [n][2] of (batch b, token t).  Returns [L_s][H][n][d] in the
    cache dtype (all source layers and heads of those tokens).
    """
    rows = np.asarray(rows, dtype=np.int64).reshape(-1, 2)
    key = stream_key(w.seed, _cache_stream(kv, turn))
    scale = torch.from_numpy(channel_scales(w)[kv])
    l = torch.arange(w.Ls).view(w.Ls, 1, 1, 1)
    h = torch.arange(w.H).view(1, w.H, 1, 1)
    b = torch.from_numpy(rows[:, 0]).view(1, 1, -1, 1)
    t = torch.from_numpy(rows[:, 1]).view(1, 1, -1, 1)
    c = torch.arange(w.d).view(1, 1, 1, w.d)
    idx = (((l * w.B + b) * w.H + h) * w.T + t) * w.d + c
    z = irwin_hall12(key, idx)
    val = z * scale.view(w.Ls, w.H, 1, w.d)
    return val.to(w.torch_dtype())


def weights(w):
    """(W [L_t][2][H][F][d], b [L_t][2][H][d]) as torch CPU tensors in the weight dtype.

    W ~ N(0, 1/F), b ~ N(0, 0.01), drawn in float64, rounded to float32 and then (bf16
    workloads) to bf16.  Index 0 of the second axis is K, 1 is V; the F rows of W are
    the k selected source layers' d channels, in ascending source-layer order.
    """
    rng = _rng(w, STREAM_W)
    W = rng.standard_normal((w.Lt, 2, w.H, w.F, w.d), dtype=np.float64) * (1.0 / np.sqrt(w.F))
    rng = _rng(w, STREAM_B)
    bias = rng.standard_normal((w.Lt, 2, w.H, w.d)) * 0.1
    Wt = torch.from_numpy(W.astype(np.float32)).to(w.torch_dtype("weight"))
    bt = torch.from_numpy(bias.astype(np.float32)).to(w.torch_dtype("weight"))
    return Wt, bt


def selection_scores(w):
    """float64 [L_t][L_s] scores from which the top-k selection is taken."""
    rng = _rng(w, STREAM_SCORES)
    if w.scores == "uniform":
        return rng.uniform(size=(w.Lt, w.Ls))
    lp = np.arange(w.Ls)[None, :] / (w.Ls - 1)
    l = np.arange(w.Lt)[:, None] / (w.Lt - 1)
    return np.exp(-((lp - l) ** 2) / (2 * 0.05 ** 2)) + 0.02 * rng.uniform(size=(w.Lt, w.Ls))


def positions(w, turn=0, lengths=None):
    """int32 [B][T] absolute positions of the mapped tokens.

    Contiguous workloads: 0..T-1 for every sequence.  Paged workload: turn j maps
    positions L0_b + T*j + [0, T) of sequence b, L0_b its initial length.
    """
    base = np.zeros(w.B, dtype=np.int64) if lengths is None else lengths + w.T * turn
    return (base[:, None] + np.arange(w.T)[None, :]).astype(np.int32)


def initial_lengths(w):
    """Paged workload: initial per-sequence lengths L0_b ~ U{lo..hi}."""
    lo, hi = w.len_range
    return _rng(w, STREAM_LENGTHS).integers(lo, hi + 1, size=w.B).astype(np.int64)


def block_table(w, pos, turn=0):
    """Paged target cache for one turn: a seeded random block table.

    Every logical block (position // block_size) that a mapped token touches gets a
    distinct physical block, in a random permutation of a pool of exactly that many
    blocks.  Returns (table int32 [B][max_blocks_per_seq] with -1 for untouched
    logical blocks, n_blocks).
    """
    pos = np.asarray(pos, dtype=np.int64)
    bs = w.block_size
    max_blocks = int(pos.max()) // bs + 1
    table = np.full((w.B, max_blocks), -1, dtype=np.int32)
    touched = [np.unique(pos[b] // bs) for b in range(w.B)]
    n_blocks = int(sum(len(t) for t in touched))
    perm = _rng(w, STREAM_BLOCKS + 1000 * turn).permutation(n_blocks).astype(np.int32)
    o = 0
    for b in range(w.B):
        table[b, touched[b]] = perm[o:o + len(touched[b])]
        o += len(touched[b])
    return table, n_blocks


def persistent_block_table(w, lengths):
    """Paged target cache that persists across every turn: one seeded random block table
    covering each sequence's final length L0_b + turns * T.

    Logical block i of sequence b (positions 16 i .. 16 i + 15) gets a distinct physical
    block, in a random permutation of a pool of exactly sum_b ceil(final_b / 16) blocks,
    including the blocks of the initial prefix that no turn maps.  Returns (table int32
    [B][max_blocks_per_seq], -1 past a sequence's last block, n_blocks)."""
    bs = w.block_size
    final = np.asarray(lengths, dtype=np.int64) + w.turns * w.T
    nb = (final + bs - 1) // bs
    table = np.full((w.B, int(nb.max())), -1, dtype=np.int32)
    n_blocks = int(nb.sum())
    perm = _rng(w, STREAM_BLOCKS + 999).permutation(n_blocks).astype(np.int32)
    o = 0
    for b in range(w.B):
        table[b, :nb[b]] = perm[o:o + nb[b]]
        o += int(nb[b])
    return table, n_blocks
