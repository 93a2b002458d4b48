"""GPU parity of budget mode (Sec. 6.5, eviction under a fixed budget)
against the oracle's BudgetTable: after every call the (key, slot, stamp)
triples of the table, and after every eviction the removed slots, the entry
count and the lookups of every key, bit-exact.  Positions are not compared
(the compaction moves kept entries; only reachability is required, and the
lookups check it)."""
import time

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_38706_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def triples(kt):
    e = kt.table.view(-1, 32).cpu().numpy()
    st = kt.stamps.cpu().numpy().view(np.uint64)
    occ = e[:, :16].any(axis=1)
    slots = e[:, 16:20].copy().view(np.uint32)[:, 0]
    assert not st[~occ].any(), "an empty entry holds a stamp"
    return sorted(zip((bytes(k) for k in e[occ, :16]), slots[occ].tolist(), st[occ].tolist()))


def _keys(rng, n):
    k = rng.integers(0, 256, (n, 32), dtype=np.uint8)
    k[:, 0] |= 1
    return k


def _batch(rng, pool, R, lo, hi):
    rows, off = [], [0]
    for _ in range(R):
        n = int(rng.integers(lo, hi))
        s = int(rng.integers(0, pool.shape[0] - n + 1))
        rows.append(pool[s:s + n])
        off.append(off[-1] + n)
    return np.ascontiguousarray(np.concatenate(rows)), np.array(off, np.int64)


def run_evict(kt, bt, budget, keep):
    ev, n_ev = kt.evict(budget, keep)
    want = bt.evict(budget, keep)
    torch.cuda.synchronize()
    kt.check("evict")
    n = int(n_ev.item())
    got = np.sort(ev[:n].cpu().numpy().view(np.uint32))
    assert n == want.size and np.array_equal(got, want)
    assert kt.entries() == len(bt)


def check_lookups(kt, bt, pool):
    off = torch.arange(0, pool.shape[0] + 1, dtype=torch.int64, device="cuda")  # one key per request
    _, slots = kt.lookup(torch.from_numpy(pool).cuda(), off)
    torch.cuda.synchronize()
    assert np.array_equal(slots.cpu().numpy().view(np.uint32), bt.table.get(pool))


@pytest.mark.parametrize("seed,log2,budget,keep", [(0, 10, 400, 300), (1, 10, 700, 700), (2, 6, 50, 20),
                                                   (3, 6, 60, 45), (4, 12, 2500, 0)])
def test_calls_and_evictions_bit_exact(seed, log2, budget, keep):
    from paper_2609_38706_gb300.service import KeyTable
    rng = np.random.default_rng(seed)
    pool = _keys(rng, min(3 * budget + 50, (1 << log2) - 1))
    kt = KeyTable(16, log2)
    kt.attach_stamps()
    bt = O.BudgetTable(1 << log2)
    slot = 0
    for call in range(12):
        if call == 0:  # a list-mode store first
            ks = pool[: min(budget, pool.shape[0])]
            sl = np.arange(slot, slot + ks.shape[0], dtype=np.uint32)
            kt.store(torch.from_numpy(ks).cuda(), sl)
            bt.store(ks, sl)
        else:
            ks, off = _batch(rng, pool, int(rng.integers(1, 40)), 1, 24)  # may cross the capacity
            sl = np.arange(slot, slot + ks.shape[0], dtype=np.uint32)
            if call % 4 == 2:
                sl[rng.random(sl.size) < 0.15] = O.NO_SLOT
            hit, slots, res, so = kt.lookup_store(torch.from_numpy(ks).cuda(), torch.from_numpy(off).cuda(), sl)
            w = bt.lookup_store(ks, off, sl)
            torch.cuda.synchronize()
            kt.take_status()  # PK_ERR_ARG (unstorable keys) and PK_ERR_TABLE_FULL are expected
            assert np.array_equal(hit.cpu().numpy(), w[0])
            assert np.array_equal(res.cpu().numpy(), w[2])
        slot += ks.shape[0]
        assert triples(kt) == bt.triples(), f"call {call}: stamps"
        run_evict(kt, bt, budget, keep)
        assert triples(kt) == bt.triples(), f"call {call}: after eviction"
        check_lookups(kt, bt, pool)
    kt.close()


def test_within_budget_changes_nothing():
    from paper_2609_38706_gb300.service import KeyTable
    rng = np.random.default_rng(5)
    kt = KeyTable(16, 10)
    kt.attach_stamps()
    keys = _keys(rng, 300)
    kt.store(torch.from_numpy(keys).cuda(), np.arange(300, dtype=np.uint32))
    before_t, before_s = kt.table.clone(), kt.stamps.clone()
    ev, n_ev = kt.evict(300, 100)
    torch.cuda.synchronize()
    kt.check()
    assert int(n_ev.item()) == 0
    assert torch.equal(kt.table, before_t) and torch.equal(kt.stamps, before_s)
    kt.close()


def test_unstamped_entries_tie():
    """Entries stored before the stamps were attached all have stamp 0 and
    are removed together."""
    from paper_2609_38706_gb300.service import KeyTable
    rng = np.random.default_rng(6)
    kt = KeyTable(16, 10)
    bt = O.BudgetTable(1 << 10)
    keys = _keys(rng, 200)
    kt.store(torch.from_numpy(keys).cuda(), np.arange(200, dtype=np.uint32))
    bt.store(keys, np.arange(200, dtype=np.uint32))
    kt.attach_stamps()
    bt.stamps.clear()
    off = np.array([0, 30], np.int64)
    kt.lookup_store(torch.from_numpy(keys[:30]).cuda(), torch.from_numpy(off).cuda(), np.full(30, O.NO_SLOT, np.uint32))
    bt.lookup_store(keys[:30], off, np.full(30, O.NO_SLOT, np.uint32))
    torch.cuda.synchronize()
    kt.take_status()
    assert triples(kt) == bt.triples()
    run_evict(kt, bt, 100, 60)
    assert len(bt) == 30
    assert triples(kt) == bt.triples()
    check_lookups(kt, bt, keys)
    kt.close()


@pytest.mark.parametrize("Wn,B", [(400, 300), (400, 370), (300, 300)])
def test_cyclic_reuse_hits_match(Wn, B):
    from paper_2609_38706_gb300.service import KeyTable
    b = 50
    rng = np.random.default_rng(Wn * 3 + B)
    pool = _keys(rng, Wn)
    kt = KeyTable(16, 11)
    kt.attach_stamps()
    bt = O.BudgetTable(1 << 11)
    slot = 0
    for call in range(4 * Wn // b):
        idx = np.arange(call * b, call * b + b) % Wn
        ks = np.ascontiguousarray(pool[idx])
        off = np.arange(0, b + 1, dtype=np.int64)
        sl = np.arange(slot, slot + b, dtype=np.uint32)
        slot += b
        hit, _, _, _ = kt.lookup_store(torch.from_numpy(ks).cuda(), torch.from_numpy(off).cuda(), sl)
        w = bt.lookup_store(ks, off, sl)
        run_evict(kt, bt, B, B)
        assert np.array_equal(hit.cpu().numpy(), w[0]), call
    assert triples(kt) == bt.triples()
    kt.close()


@pytest.mark.parametrize("name", ["multi_adapter", "small_block"])
def test_workload_step_with_budget(name):
    """A workload's seeded table, one lookup-and-store of its batch, then an
    eviction to half the entries (reduced size: every entry compared)."""
    from paper_2609_38706_gb300.service import KeyTable
    wl = W.reduced(name)
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    kt.attach_stamps()
    d = kt.digests(wl.descriptors)
    pko, pkeys = kt.derive(wl.prior.tokens, wl.prior.tok_off, wl.prior.desc_idx, d)
    pko_h = pko.cpu().numpy()
    seed_keys = W.seed_list(pkeys.cpu().numpy()[: int(pko_h[-1])], pko_h, wl.prior_chunks)
    kt.seed(seed_keys, wl.filler, wl.target_entries)
    bt = O.BudgetTable(wl.capacity)
    if seed_keys.shape[0]:  # KeyTable.seed makes no store call for an empty seed list
        bt.store(seed_keys, np.arange(seed_keys.shape[0], dtype=np.uint32))
    need = wl.target_entries - len(bt)
    if need > 0:
        bt.store(wl.filler[:need], np.arange(seed_keys.shape[0], seed_keys.shape[0] + need, dtype=np.uint32))
    assert triples(kt) == bt.triples()
    key_off, keys = kt.derive(wl.batch.tokens, wl.batch.tok_off, wl.batch.desc_idx, d)
    N = int(key_off[-1])
    sl = np.arange(N, dtype=np.uint32) + 10_000_000
    kt.lookup_store(keys, key_off, sl)
    bt.lookup_store(keys.cpu().numpy()[:N], key_off.cpu().numpy(), sl)
    torch.cuda.synchronize()
    kt.check("lookup_store")
    assert triples(kt) == bt.triples()
    half = len(bt) // 2
    run_evict(kt, bt, half, half)
    assert triples(kt) == bt.triples()
    check_lookups(kt, bt, np.ascontiguousarray(keys.cpu().numpy()[:N]))
    kt.close()


def test_all_stamps_equal():
    """Every stamp 0 (stored before the stamps were attached): the (keep+1)-th
    largest is 0 and every entry goes."""
    from paper_2609_38706_gb300.service import KeyTable
    rng = np.random.default_rng(10)
    kt = KeyTable(16, 11)
    bt = O.BudgetTable(1 << 11)
    keys = _keys(rng, 900)
    kt.store(torch.from_numpy(keys).cuda(), np.arange(900, dtype=np.uint32))
    bt.table.store(keys, np.arange(900, dtype=np.uint32))
    kt.attach_stamps()
    run_evict(kt, bt, 500, 100)
    assert len(bt) == 0 and kt.entries() == 0
    assert not kt.table.any()
    kt.close()


def test_large_table_sampled():
    """2^20 entries, 600k stored by two list-mode calls and a lookup-and-store,
    evicted to 200k: removed slots compared in full, kept entries as a set,
    lookups of a sample."""
    from paper_2609_38706_gb300.service import KeyTable
    rng = np.random.default_rng(11)
    log2 = 20
    kt = KeyTable(16, log2)
    kt.attach_stamps()
    bt = O.BudgetTable(1 << log2)
    keys = _keys(rng, 600_000)
    for a, b in ((0, 300_000), (300_000, 600_000)):
        sl = np.arange(a, b, dtype=np.uint32)
        kt.store(torch.from_numpy(keys[a:b]).cuda(), sl)
        bt.store(keys[a:b], sl)
    reuse = np.ascontiguousarray(keys[rng.permutation(600_000)[:50_000]])  # touch 50k of them again
    off = np.arange(0, 50_001, 10, dtype=np.int64)
    sl = np.arange(50_000, dtype=np.uint32) + 10_000_000
    kt.lookup_store(torch.from_numpy(reuse).cuda(), torch.from_numpy(off).cuda(), sl)
    bt.lookup_store(reuse, off, sl)
    torch.cuda.synchronize()
    kt.check("lookup_store")
    run_evict(kt, bt, 500_000, 200_000)
    assert triples(kt) == bt.triples()
    check_lookups(kt, bt, np.ascontiguousarray(keys[rng.integers(0, 600_000, 20_000)]))
    kt.close()


def test_barrier_wait_runs_out_and_the_context_stays_usable():
    """The bounded grid barrier of pk_evict: one CTA withholds its arrival at
    the first barrier (a flag that nothing sets), the other CTAs' waits run
    out after a short bound, the launch ends by itself with PK_ERR_TIMEOUT,
    the table and stamps are untouched (the first barrier precedes every
    write), and the next calls on the context work and match the oracle."""
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300.service import KeyTable
    log2 = 14
    rng = np.random.default_rng(11)
    pool = _keys(rng, 6000)
    kt = KeyTable(16, log2)
    kt.attach_stamps()
    bt = O.BudgetTable(1 << log2)
    sl = np.arange(pool.shape[0], dtype=np.uint32)
    kt.store(torch.from_numpy(pool).cuda(), sl)
    bt.store(pool, sl)
    torch.cuda.synchronize()
    kt.check("store")
    table0, stamps0 = kt.table.clone(), kt.stamps.clone()
    t0 = time.perf_counter()
    pk.pk_evict_barrier_timeout_test(kt.ctx, 4000, kt.evict_scratch, 1 << 12, kt.status)
    torch.cuda.synchronize()
    took = time.perf_counter() - t0
    assert kt.take_status() == pk.PK_ERR_TIMEOUT
    assert took < 5.0
    assert torch.equal(kt.table, table0) and torch.equal(kt.stamps, stamps0)
    run_evict(kt, bt, 4000, 3000)  # the same eviction, now with every CTA arriving
    assert triples(kt) == bt.triples()
    check_lookups(kt, bt, pool)
    kt.close()
