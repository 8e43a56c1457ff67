"""Host logic of the per-head tensor-core kernel's source-tile schedule (no GPU).

The gather of Sec. 3.2 reads the k selected source layers of every target layer.  The
per-head tensor-core kernel keeps up to four source tiles of a token tile in tensor
memory; `kvx_tc_load_schedule` returns the schedule `kvx_create` builds for it.  Checked
here against what fixes it independently of its code:
 * the number of loads per token tile is the minimum over every eviction choice
   (exhaustive search over the resident sets, small cases);
 * on every synthetic workload each selected source layer is loaded once per token tile,
   which is the kernel's algorithmic source traffic;
 * a simulation of the kernel's three parties over several token tiles: the prologue
   (loads in schedule order; before a load it waits for the releases the load word names)
   and the two issuers (target layers l with l % 2 == i; first use of a tile waits for
   its load, last use releases the slot).  Every wait is an mbarrier parity wait, as on
   the device.  Random and adversarial interleavings must end with every use reading the
   tile of its selected layer, no wait blocked forever, and no barrier completing a phase
   while its waiter still has an earlier phase to consume (a parity wait would then
   alias the two phases).
"""
import random

import numpy as np
import pytest

from paper_2608_03893_gb300 import build as kbuild
from paper_2608_03893_gb300 import kvx
from paper_2608_03893_gb300 import synthetic as syn

SLOTS = 4


@pytest.fixture(scope="module", autouse=True)
def built():
    kbuild.build()
    kvx.lib()


def min_loads(seq, capacity=SLOTS):
    """Fewest loads that serve the use sequence `seq` with `capacity` resident tiles,
    starting empty: exhaustive search over every eviction choice."""
    best = {frozenset(): 0}
    for x in seq:
        nxt = {}
        for state, cost in best.items():
            if x in state:
                cand = [(state, cost)]
            elif len(state) < capacity:
                cand = [(state | {x}, cost + 1)]
            else:
                cand = [((state - {v}) | {x}, cost + 1) for v in state]
            for st, c in cand:
                if c < nxt.get(st, 1 << 30):
                    nxt[st] = c
        best = nxt
    return min(best.values())


class Barrier:
    """An mbarrier seen through parity waits: `done` phases completed; its one waiter
    has consumed `seen` of them."""

    def __init__(self):
        self.done = 0
        self.seen = 0
        self.payload = []

    def complete(self, what, item=None):
        # the waiter must have consumed every completed phase, or its next parity wait
        # could not tell phase n from phase n + 2
        assert self.done == self.seen, "%s: a phase completed while its waiter was %d behind" % (
            what, self.done - self.seen)
        self.done += 1
        self.payload.append(item)

    def ready(self):
        n = self.seen
        return (self.done & 1) != (n & 1)     # try_wait.parity(n & 1)

    def consume(self):
        item = self.payload[self.seen]
        self.seen += 1
        return item


def simulate(sel, layer, word, use, units, pick):
    Lt, k = sel.shape
    tready = [[Barrier() for _ in range(2)] for _ in range(SLOTS)]
    tfree = [[Barrier() for _ in range(2)] for _ in range(SLOTS)]
    slot_layer = [-1] * SLOTS
    slot_serial = [-1] * SLOTS
    counters = {"serial": 0, "uses": 0}

    def prologue():
        loaded = [False] * SLOTS
        for _ in range(units):
            for e in range(len(layer)):
                lw = int(word[e])
                s = lw & 3
                if loaded[s]:
                    for i in range(2):
                        if (lw >> (2 + i)) & 1:
                            yield tfree[s][i]
                            tfree[s][i].consume()
                loaded[s] = True
                counters["serial"] += 1
                slot_layer[s] = int(layer[e])
                slot_serial[s] = counters["serial"]
                for i in range(2):
                    if (lw >> (4 + i)) & 1:
                        tready[s][i].complete("tready[%d][%d]" % (s, i), counters["serial"])

    def issuer(i):
        held = [-1] * SLOTS
        for _ in range(units):
            for l in range(i, Lt, 2):
                for j in range(k):
                    f = int(use[l][j])
                    s = f & 3
                    if f & 4:
                        yield tready[s][i]
                        held[s] = tready[s][i].consume()
                    assert held[s] == slot_serial[s], "use (%d, %d): its tile was overwritten" % (l, j)
                    assert slot_layer[s] == sel[l][j], "use (%d, %d) reads layer %d, selected %d" % (
                        l, j, slot_layer[s], sel[l][j])
                    counters["uses"] += 1
                    if f & 16:
                        tfree[s][i].complete("tfree[%d][%d]" % (s, i))

    actors = [prologue(), issuer(0), issuer(1)]
    waiting = [None] * 3
    live = [True] * 3

    def step(a):
        try:
            waiting[a] = next(actors[a])
        except StopIteration:
            live[a] = False
            waiting[a] = None

    for a in range(3):
        step(a)
    while any(live):
        runnable = [a for a in range(3) if live[a] and (waiting[a] is None or waiting[a].ready())]
        assert runnable, "deadlock: every live party waits"
        step(pick(runnable))
    assert counters["uses"] == units * Lt * k
    return counters["serial"]


def random_selection(rng, Ls, Lt, k, sort):
    rows = []
    for _ in range(Lt):
        r = rng.sample(range(Ls), k)
        rows.append(sorted(r) if sort else r)
    return np.array(rows, dtype=np.int32)


def pickers(rng):
    return {
        "random": lambda r: rng.choice(r),
        "prologue first": lambda r: r[0],
        "issuers first": lambda r: r[-1],
        "issuer 1 first": lambda r: 2 if 2 in r else r[0],
    }


def test_loads_are_the_minimum_over_every_eviction_choice():
    rng = random.Random(11)
    for trial in range(300):
        k = rng.randint(1, 4)
        Ls = rng.randint(k, 8)
        Lt = rng.randint(1, 7)
        sel = random_selection(rng, Ls, Lt, k, sort=trial % 2 == 0)
        layer, word, use = kvx.kvx_tc_load_schedule(sel, Ls)
        assert len(layer) == min_loads(sel.reshape(-1).tolist()), (sel.tolist(), layer.tolist())


def test_every_selected_layer_is_loaded_once_on_the_workloads():
    for name in syn.WORKLOADS:
        w = syn.workload(name)
        if w.k > SLOTS:
            continue
        sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
        layer, word, use = kvx.kvx_tc_load_schedule(sel, w.Ls)
        assert sorted(layer.tolist()) == sorted(set(sel.reshape(-1).tolist())), name


def test_shared_layers_and_a_single_layer():
    # every target layer selects the same k layers: k loads, each used by both issuers
    sel = np.tile(np.arange(4, dtype=np.int32), (9, 1))
    layer, word, use = kvx.kvx_tc_load_schedule(sel, 6)
    assert layer.tolist() == [0, 1, 2, 3]
    assert all((w >> 4) & 3 == 3 for w in word)
    # one target layer, one source layer: one load, one use that waits and releases
    layer, word, use = kvx.kvx_tc_load_schedule(np.array([[3]], dtype=np.int32), 5)
    assert layer.tolist() == [3] and use.tolist() == [[(word[0] & 3) | 4 | 16]]


@pytest.mark.parametrize("seed", range(4))
def test_protocol_simulation(seed):
    rng = random.Random(seed)
    for trial in range(120):
        k = rng.randint(1, 4)
        Ls = rng.randint(k, 12)
        Lt = rng.randint(1, 13)
        sel = random_selection(rng, Ls, Lt, k, sort=trial % 3 != 0)
        layer, word, use = kvx.kvx_tc_load_schedule(sel, Ls)
        for pname, pick in pickers(rng).items():
            loads = simulate(sel, layer, word, use, units=3, pick=pick)
            assert loads == 3 * len(layer), pname


def test_protocol_simulation_on_the_workloads():
    rng = random.Random(5)
    for name in ("qwen3_14b_32b_t32768_k4", "qwen3_14b_32b_t32768_k1", "llama31_8b_70b_b4x8192_k3",
                 "llama31_70b_8b_b4x8192_k3", "qwen3_32b_14b_paged_b16_turn2048_k4"):
        w = syn.workload(name)
        sel = kvx.kvx_select_topk(syn.selection_scores(w), w.k)
        layer, word, use = kvx.kvx_tc_load_schedule(sel, w.Ls)
        for pick in pickers(rng).values():
            simulate(sel, layer, word, use, units=2, pick=pick)


def test_simulation_catches_a_missing_release_wait():
    # the check is live: drop issuer 0's release bit from one load word (a schedule that
    # overwrites a tile before issuer 0 has finished with it) and the simulation fails
    rng = random.Random(3)
    for _ in range(200):
        sel = random_selection(rng, 10, 8, 3, sort=True)
        layer, word, use = kvx.kvx_tc_load_schedule(sel, 10)
        victims = [e for e in range(len(word)) if (word[e] >> 2) & 1 and e >= SLOTS]
        if victims:
            break
    bad = word.copy()
    bad[victims[0]] &= ~(1 << 2)
    failed = 0
    for pick in pickers(rng).values():
        try:
            simulate(sel, layer, bad, use, units=2, pick=pick)
        except AssertionError:
            failed += 1
    assert failed >= 1


def test_rejects_bad_tables():
    ok = np.array([[0, 1], [1, 2]], dtype=np.int32)
    kvx.kvx_tc_load_schedule(ok, 3)
    for sel, Ls, status in (
            (np.array([[0, 0], [1, 2]], dtype=np.int32), 3, kvx.KVX_ERR_INVALID_ARG),   # repeated layer
            (np.array([[0, 3], [1, 2]], dtype=np.int32), 3, kvx.KVX_ERR_INVALID_ARG),   # out of range
            (np.array([[0, -1], [1, 2]], dtype=np.int32), 3, kvx.KVX_ERR_INVALID_ARG),
            (np.arange(5, dtype=np.int32)[None, :], 6, kvx.KVX_ERR_UNSUPPORTED),        # k > 4
            (np.array([[0, 1, 2]], dtype=np.int32), 2, kvx.KVX_ERR_INVALID_ARG)):       # k > L_s
        with pytest.raises(kvx.KvxError) as e:
            kvx.kvx_tc_load_schedule(sel, Ls)
        assert e.value.status == status, sel.tolist()
