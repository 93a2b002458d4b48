"""Pins of the oracle's eviction under a fixed budget (Sec. 6.5): the
stamp-and-threshold formulation against an independent one (a recency list
that moves each used key to its end, popped from the front), invariants of
one eviction, the tie rule, and the thrashing the paper reports as a closed
form (a cyclic reuse pattern under LRU hits nothing once the working set
exceeds the budget, and everything after the first pass when it fits)."""
from collections import OrderedDict

import numpy as np
import pytest

import oracle as O


def _keys(rng, n):
    k = rng.integers(0, 256, (n, 32), dtype=np.uint8)
    k[:, 0] |= 1
    return k


class RecencyList:
    """Sequential LRU: in each call the keys are used in index order (a used
    key moves to the end); eviction pops from the front down to `keep`."""

    def __init__(self):
        self.od: OrderedDict[bytes, int] = OrderedDict()

    def lookup_store(self, keys, key_off, new_slots):
        p = O.prefix128(keys)
        present0 = [p[e].tobytes() in self.od for e in range(p.shape[0])]
        # the table effect: lookup (first miss) then store the miss ranges in order
        for r in range(len(key_off) - 1):
            a, b = int(key_off[r]), int(key_off[r + 1])
            h = next((j for j in range(b - a) if not present0[a + j]), b - a)
            for e in range(a + h, b):
                k = p[e].tobytes()
                if k not in self.od and int(new_slots[e]) != O.NO_SLOT:
                    self.od[k] = int(new_slots[e])
        for e in range(p.shape[0]):  # uses, in index order
            k = p[e].tobytes()
            if present0[e] or (int(new_slots[e]) != O.NO_SLOT and k in self.od):
                self.od.move_to_end(k)

    def evict(self, budget, keep):
        out = []
        if len(self.od) > budget:
            while len(self.od) > keep:
                out.append(self.od.popitem(last=False)[1])
        return np.array(sorted(out), np.uint32)


def _batch(rng, pool, R, lo, hi):
    rows, off = [], [0]
    for _ in range(R):
        n = int(rng.integers(lo, hi))
        start = int(rng.integers(0, pool.shape[0] - n + 1))
        rows.append(pool[start:start + n])
        off.append(off[-1] + n)
    return np.concatenate(rows) if rows else pool[:0], np.array(off, np.int64)


@pytest.mark.parametrize("seed", range(6))
def test_stamps_match_a_recency_list(seed):
    rng = np.random.default_rng(seed)
    pool = _keys(rng, 300)
    bt, rl = O.BudgetTable(1 << 10), RecencyList()
    budget, keep = 150, 120
    slot = 0
    for call in range(25):
        keys, off = _batch(rng, pool, int(rng.integers(1, 8)), 1, 30)
        new_slots = np.arange(slot, slot + keys.shape[0], dtype=np.uint32)
        slot += keys.shape[0]
        if call % 5 == 3:  # some keys not storable
            new_slots[rng.random(keys.shape[0]) < 0.2] = O.NO_SLOT
        bt.lookup_store(keys, off, new_slots)
        rl.lookup_store(keys, off, new_slots)
        assert sorted(bt.table.map.items()) == sorted(rl.od.items())
        ev_b, ev_r = bt.evict(budget, keep), rl.evict(budget, keep)
        assert np.array_equal(ev_b, ev_r), call
        assert sorted(bt.table.map.items()) == sorted(rl.od.items())


def test_one_eviction_invariants():
    rng = np.random.default_rng(7)
    bt = O.BudgetTable(1 << 12)
    keys = _keys(rng, 2000)
    off = np.arange(0, 2001, 10, dtype=np.int64)
    bt.lookup_store(keys, off, np.arange(2000, dtype=np.uint32))
    before = dict(bt.table.map)
    stamps = dict(bt.stamps)
    ev = bt.evict(1500, 1000)
    assert len(bt) == 1000 and ev.size == 1000
    assert sorted(list(bt.table.map.values()) + ev.tolist()) == sorted(before.values())
    kept = [stamps[k] for k in bt.table.map]
    gone = [stamps[k] for k in before if k not in bt.table.map]
    assert min(kept) > max(gone)
    # within the budget nothing happens; keep == 0 empties the table
    assert bt.evict(1000, 500).size == 0 and len(bt) == 1000
    assert bt.evict(999, 0).size == 1000 and len(bt) == 0


def test_unstamped_entries_tie_and_go_together():
    rng = np.random.default_rng(8)
    bt = O.BudgetTable(1 << 10)
    keys = _keys(rng, 100)
    bt.table.store(keys, np.arange(100, dtype=np.uint32))  # not through the budget table: stamp 0
    off = np.array([0, 10], np.int64)
    bt.lookup_store(keys[:10], off, np.full(10, O.NO_SLOT, np.uint32))  # uses 10 of them
    ev = bt.evict(50, 40)
    assert ev.size == 90 and len(bt) == 10  # the 90 zero stamps tie below the 40th largest
    assert sorted(bt.table.map.values()) == list(range(10))


def test_stamp_is_call_number_and_index():
    rng = np.random.default_rng(9)
    bt = O.BudgetTable(1 << 8)
    k = _keys(rng, 4)
    bt.store(k[:2], np.array([5, 6], np.uint32))                      # call 1
    bt.lookup_store(k[[1, 2, 1]], np.array([0, 3]), np.array([7, 8, 9], np.uint32))  # call 2
    st = {kk[:4]: v for kk, _, v in bt.triples()}
    p = O.prefix128(k)
    assert st[p[0].tobytes()[:4]] == (1 << 32) | 0
    assert st[p[1].tobytes()[:4]] == (2 << 32) | 2                    # last use: index 2 of call 2
    assert st[p[2].tobytes()[:4]] == (2 << 32) | 1


@pytest.mark.parametrize("W,B", [(400, 300), (400, 350), (400, 399), (450, 420), (200, 300), (300, 300)])
def test_cyclic_reuse_thrashes_once_the_working_set_exceeds_the_budget(W, B):
    """W distinct chunks requested cyclically, b = 50 per call, evicting to B
    after every call.  At the start of a call the table holds the keys of
    the last B uses, and the j-th key of the call was last used W - j uses
    before the call started, so it hits iff j >= W - B: b - (W - B) hits per
    call, clamped to [0, b].  All hit when W <= B; none once W >= B + b,
    the thrashing of LRU under cyclic reuse."""
    b = 50
    rng = np.random.default_rng(W + B)
    pool = _keys(rng, W)
    bt = O.BudgetTable(1 << 11)
    hits = total = 0
    slot = 0
    calls = 4 * W // b
    for call in range(calls):
        idx = np.arange(call * b, call * b + b) % W
        off = np.arange(0, b + 1, dtype=np.int64)  # one chunk per request
        hit, _, _, _ = bt.lookup_store(pool[idx], off, np.arange(slot, slot + b, dtype=np.uint32))
        slot += b
        bt.evict(B, B)
        if call >= -(-W // b):  # after the first pass
            hits += int(hit.sum())
            total += b
    per_call = min(max(b - (W - B), 0), b)
    assert hits == per_call * (total // b)
