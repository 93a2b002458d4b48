"""Pins for the oracle's table semantics (lookup / store / seeding).

DictTable is the plain definition (a Python dict, array-order inserts);
SortedTable must agree with it everywhere.  Closed forms: the Tiny
configuration's generator-known hit lengths, the provenance sweep's 16*D
distinct prefix keys (storage linear in provenance diversity, Sec. 6.5), and
h_r = n_r for every request after its misses are stored.
"""
import numpy as np
import pytest

import oracle as O
from paper_2609_38706_gb300 import workloads as W


def _rand_keys(rng, n, pool):
    base = rng.integers(0, 256, (pool, 32), dtype=np.uint8)
    return base[rng.integers(0, pool, n)]


@pytest.mark.parametrize("seed", range(20))
def test_sorted_matches_dict(seed):
    rng = np.random.default_rng(seed)
    cap = 1 << int(rng.integers(3, 8))
    td, ts = O.DictTable(cap), O.SortedTable(cap)
    for _ in range(4):
        n = int(rng.integers(0, 3 * cap))
        keys = _rand_keys(rng, n, max(cap, 1))
        if n and rng.random() < 0.3:
            keys[rng.integers(0, n), :16] = 0                      # reserved key
        slots = rng.integers(0, 1 << 32, n, dtype=np.uint64).astype(np.uint32)
        if n and rng.random() < 0.3:
            slots[rng.integers(0, n)] = O.NO_SLOT                  # invalid slot value
        rd, sd = td.store(keys, slots)
        rs, ss = ts.store(keys, slots)
        assert np.array_equal(rd, rs) and np.array_equal(sd, ss)
        assert len(td) == len(ts) <= cap - 1
        q = _rand_keys(rng, 50, max(cap, 1))
        assert np.array_equal(td.get(q), ts.get(q))


def test_first_occurrence_wins_and_present_keeps_slot():
    t = O.DictTable(16)
    k = np.zeros((4, 32), np.uint8)
    k[:, 0] = [1, 2, 1, 3]
    res, so = t.store(k, np.array([10, 11, 12, 13]))
    assert res.tolist() == [O.STORE_INSERTED, O.STORE_INSERTED, O.STORE_PRESENT, O.STORE_INSERTED]
    assert so.tolist() == [10, 11, 10, 13]
    res, so = t.store(k[:1], np.array([99]))
    assert res.tolist() == [O.STORE_PRESENT] and so.tolist() == [10]


def test_capacity_keeps_one_empty_slot():
    t = O.DictTable(8)
    k = np.zeros((10, 32), np.uint8)
    k[:, 0] = np.arange(1, 11)
    res, _ = t.store(k, np.arange(10))
    assert (res == O.STORE_INSERTED).sum() == 7
    assert res[7:].tolist() == [O.PK_ERR_TABLE_FULL] * 3


def test_bad_capacity():
    for cap in (0, 1, 3, 12):
        with pytest.raises(O.OracleError):
            O.DictTable(cap)


def test_lookup_first_miss_ends_prefix():
    t = O.DictTable(64)
    k = np.zeros((5, 32), np.uint8)
    k[:, 0] = np.arange(1, 6)
    t.store(k[[0, 1, 3, 4]], np.arange(4))
    hit, slots = O.lookup(t, k, np.array([0, 5]))
    assert hit.tolist() == [2]                     # chunk 2 missing: later hits do not extend h
    assert slots.tolist() == [0, 1, O.NO_SLOT, 2, 3]


def _seeded(wl, table_cls):
    d = O.descriptor_digests(wl.descriptors)
    C = wl.chunk_tokens
    pko, pk = O.derive_keys(wl.prior.tokens, wl.prior.tok_off, C, wl.prior.desc_idx, d)
    seeds = W.seed_list(pk, pko, wl.prior_chunks)
    t = O.seed_table(table_cls(wl.capacity), seeds, wl.filler, wl.target_entries)
    ko, keys = O.derive_keys(wl.batch.tokens, wl.batch.tok_off, C, wl.batch.desc_idx, d)
    return t, ko, keys, seeds


def test_tiny_generator_known_hits():
    wl = W.tiny()
    t, ko, keys, seeds = _seeded(wl, O.DictTable)
    assert len(t) == wl.target_entries == 16 and seeds.shape[0] == 8
    hit, slots = O.lookup(t, keys, ko)
    assert hit.tolist() == wl.expected_hits.tolist() == [2, 2, 2, 2, 0, 2, 0, 0]
    # request 5 repeats request 1 -> the slots stored for request 1's keys (seed positions 2, 3)
    assert slots[ko[5]:ko[6]].tolist() == [2, 3]


@pytest.mark.parametrize("D", [1, 4, 16])
def test_sweep_storage_linear_in_diversity(D):
    wl = W.reduced(f"provenance_sweep_D{D}")
    d = O.descriptor_digests(wl.descriptors)
    pko, pk = O.derive_keys(wl.prior.tokens, wl.prior.tok_off, wl.chunk_tokens, wl.prior.desc_idx, d)
    per_prefix = 1024 // wl.chunk_tokens
    distinct = {bytes(x) for x in O.prefix128(pk)}
    assert len(distinct) == per_prefix * D
    t, ko, keys, _ = _seeded(wl, O.SortedTable)
    hit, _ = O.lookup(t, keys, ko)
    n = np.diff(ko)
    assert np.array_equal(hit, np.minimum(n, per_prefix))


def test_long_context_half_hits():
    wl = W.long_context(R=6, T=4096, n_shared=3, shared_len=2048, capacity_log2=10)
    t, ko, keys, _ = _seeded(wl, O.DictTable)
    hit, _ = O.lookup(t, keys, ko)
    assert hit.tolist() == wl.expected_hits.tolist() == [8] * 6


@pytest.mark.parametrize("name", ["multi_adapter", "small_block", "long_context"])
def test_store_misses_then_all_hit(name):
    wl = W.reduced(name)
    for cls in (O.DictTable, O.SortedTable):
        t, ko, keys, _ = _seeded(wl, cls)
        before = len(t)
        hit, _ = O.lookup(t, keys, ko)
        slots = np.arange(keys.shape[0], dtype=np.uint32) + 10_000_000
        res, so = O.store_misses(t, keys, ko, hit, slots)
        n_new = int((res == O.STORE_INSERTED).sum())
        assert len(t) == before + n_new
        assert not np.any(res < 0)
        hit2, slots2 = O.lookup(t, keys, ko)
        assert np.array_equal(hit2, np.diff(ko))
        stored = res > 0
        assert np.array_equal(slots2[stored], so[stored])


def test_sorted_and_dict_seed_identically():
    wl = W.reduced("small_block")
    td, ko, keys, _ = _seeded(wl, O.DictTable)
    ts, _, _, _ = _seeded(wl, O.SortedTable)
    assert len(td) == len(ts)
    assert np.array_equal(td.get(keys), ts.get(keys))
    assert np.array_equal(td.get(wl.filler[:100]), ts.get(wl.filler[:100]))
