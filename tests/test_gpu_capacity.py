"""GPU parity of the store at the capacity threshold (Sec. 2.1: a miss
computes and writes new state; the table keeps at most capacity - 1 entries so
that every probe meets an empty entry).

The oracle's DictTable processes a store call's entries one at a time in
index order and refuses a new key once the table would reach capacity.  Every
call here crosses that threshold, on tables of 2^3 to 2^12 entries, with heavy
in-batch duplicates, reserved keys and unstorable slots mixed in, in every
mode that inserts: pk_store in list and range mode (per-request and per-key
kernels), pk_lookup_store (one warp per request, work-taking warps, per-key
kernels), pk_derive_lookup_store, budget mode, and pk_store_noalloc.  After
every call: each result and output slot equals the oracle's, element by
element; the table holds exactly the oracle's (key, slot) pairs; and at least
one entry is empty."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_38706_gb300 import pk
from paper_2609_38706_gb300 import workloads as W

pytestmark = pytest.mark.gpu

LOG2S = [3, 4, 5, 6, 7, 8, 9, 10, 11, 12]


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def KT(log2, C=16, max_probe=0):
    from paper_2609_38706_gb300.service import KeyTable
    return KeyTable(C, log2, max_probe)


def pairs(table: torch.Tensor):
    e = table.view(-1, 32).cpu().numpy()
    occ = e[:, :16].any(axis=1)
    slots = e[:, 16:20].copy().view(np.uint32)[:, 0]
    return sorted(zip((bytes(k) for k in e[occ, :16]), slots[occ].tolist()))


def empty_entries(table: torch.Tensor) -> int:
    return int((~table.view(-1, 32)[:, :16].bool().any(dim=1)).sum().item())


def check_table(kt_table: torch.Tensor, dt: O.DictTable, where: str):
    assert pairs(kt_table) == sorted(dt.map.items()), f"{where}: table contents"
    assert empty_entries(kt_table) >= 1, f"{where}: no empty entry left"


def pool_keys(rng, n, same_home_frac=0.25):
    """n distinct 32-byte keys, none with an all-zero prefix; a fraction share
    their first 8 bytes (one home entry) so that clusters form."""
    k = rng.integers(0, 256, (n, 32), dtype=np.uint8)
    k[:, 0] |= 1
    m = int(n * same_home_frac)
    if m:
        k[:m, :8] = k[0, :8]
        k[:m, 8:12] = np.arange(m, dtype=np.uint32).view(np.uint8).reshape(m, 4)
    return np.ascontiguousarray(k)


def draw(rng, pool, n, dup_frac):
    """n keys from the pool: a fresh run with in-batch repeats of its own
    earlier keys (dup_frac of the entries)."""
    idx = rng.integers(0, pool.shape[0], n)
    rep = rng.random(n) < dup_frac
    for i in np.nonzero(rep)[0]:
        if i:
            idx[i] = idx[int(rng.integers(0, i))]
    return np.ascontiguousarray(pool[idx])


def to_dev(a, dtype=torch.int32):
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda", dtype=dtype) if dtype != torch.uint8 else \
        torch.from_numpy(np.ascontiguousarray(a)).cuda()


def u32(t):
    return t.cpu().numpy().view(np.uint32)


def sprinkle(rng, keys, slots, frac=0.03):
    """A few reserved (all-zero prefix) keys and unstorable slots."""
    keys = keys.copy()
    slots = slots.copy()
    z = rng.random(keys.shape[0]) < frac
    keys[z, :16] = 0
    bad = rng.random(keys.shape[0]) < frac
    slots[bad] = O.NO_SLOT
    return keys, slots


# ---------------------------------------------------------------------------
# list mode
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("log2", LOG2S)
def test_list_mode_crossing_capacity(log2):
    cap = 1 << log2
    rng = np.random.default_rng(100 + log2)
    pool = pool_keys(rng, 2 * cap + 5)
    kt = KT(log2)
    dt = O.DictTable(cap)
    slot = 0
    refused = 0
    for call in range(7):
        n = int(rng.integers(max(1, cap // 4), 2 * cap + 1))
        keys = draw(rng, pool, n, dup_frac=(0.0, 0.3, 0.8)[call % 3])
        slots = np.arange(slot, slot + n, dtype=np.uint32)
        if call % 2:
            keys, slots = sprinkle(rng, keys, slots)
        slot += n
        res, so = kt.store(to_dev(keys, torch.uint8), to_dev(slots))
        want_res, want_so = dt.store(keys, slots)
        st = kt.take_status()
        assert np.array_equal(res.cpu().numpy(), want_res), f"log2 {log2} call {call}: results"
        assert np.array_equal(u32(so), want_so), f"log2 {log2} call {call}: output slots"
        assert kt.entries() == len(dt)
        check_table(kt.table, dt, f"log2 {log2} call {call}")
        errs = want_res[want_res < 0]
        assert (st == 0) == (errs.size == 0) and (st == 0 or st in set(errs.tolist()))
        refused += int((want_res == O.PK_ERR_TABLE_FULL).sum())
    assert refused > 0 and len(dt) == cap - 1  # the calls filled the table
    kt.close()


@pytest.mark.parametrize("log2", [6, 10, 12])
def test_deferred_keys_that_all_fit(log2):
    """entries + n >= capacity but the call's new keys fit: the deferred keys
    are claimed in parallel; nothing is refused."""
    cap = 1 << log2
    rng = np.random.default_rng(7 + log2)
    pool = pool_keys(rng, cap)
    kt = KT(log2)
    dt = O.DictTable(cap)
    first = pool[: cap // 2]
    s0 = np.arange(first.shape[0], dtype=np.uint32)
    kt.store(to_dev(first, torch.uint8), to_dev(s0))
    dt.store(first, s0)
    # mostly keys already present, repeated, plus a few new ones (also repeated)
    idx = np.concatenate([rng.integers(0, cap // 2, cap), cap // 2 + rng.integers(0, 9, 40)])
    rng.shuffle(idx)
    keys = np.ascontiguousarray(pool[idx])
    slots = np.arange(1000, 1000 + keys.shape[0], dtype=np.uint32)
    res, so = kt.store(to_dev(keys, torch.uint8), to_dev(slots))
    want_res, want_so = dt.store(keys, slots)
    kt.check("store")
    assert (want_res != O.PK_ERR_TABLE_FULL).all()
    assert np.array_equal(res.cpu().numpy(), want_res)
    assert np.array_equal(u32(so), want_so)
    check_table(kt.table, dt, "fit")
    kt.close()


def test_full_table_refuses_every_new_key_in_order():
    """One empty entry left: the first new key of a call is refused, and a
    duplicate of a refused key is refused too."""
    cap = 16
    rng = np.random.default_rng(3)
    pool = pool_keys(rng, 40, same_home_frac=0.5)
    kt = KT(4)
    dt = O.DictTable(cap)
    for call in range(4):
        keys = np.ascontiguousarray(pool[rng.integers(0, 40, 30)])
        slots = rng.integers(0, 2**31, 30).astype(np.uint32)
        res, so = kt.store(to_dev(keys, torch.uint8), to_dev(slots))
        want_res, want_so = dt.store(keys, slots)
        kt.take_status()
        assert np.array_equal(res.cpu().numpy(), want_res)
        assert np.array_equal(u32(so), want_so)
        check_table(kt.table, dt, f"call {call}")
    kt.close()


# ---------------------------------------------------------------------------
# range mode and lookup-and-store
# ---------------------------------------------------------------------------
def requests(rng, pool, R, lo, hi, dup_frac=0.3):
    """R requests of lo..hi-1 keys, each a run of the pool (shared prefixes
    between requests) with some repeats."""
    rows, off = [], [0]
    for _ in range(R):
        n = int(rng.integers(lo, hi))
        s = int(rng.integers(0, max(1, pool.shape[0] - n)))
        row = pool[s:s + n].copy()
        rep = rng.random(row.shape[0]) < dup_frac
        for i in np.nonzero(rep)[0]:
            row[i] = pool[int(rng.integers(0, pool.shape[0]))]
        rows.append(row)
        off.append(off[-1] + row.shape[0])
    keys = np.ascontiguousarray(np.concatenate(rows)) if rows else np.zeros((0, 32), np.uint8)
    return keys, np.array(off, np.int64)


# (R, lo, hi): many short requests (one warp per request), few long requests
# (one warp per 32 keys)
SHAPES = [(40, 1, 9), (1100, 0, 4), (3, 100, 400)]


@pytest.mark.parametrize("log2", [3, 5, 8, 10, 12])
@pytest.mark.parametrize("shape", SHAPES)
def test_range_mode_crossing_capacity(log2, shape):
    R, lo, hi = shape
    cap = 1 << log2
    rng = np.random.default_rng(log2 * 31 + R)
    pool = pool_keys(rng, 2 * cap + 40)
    kt = KT(log2)
    dt = O.DictTable(cap)
    slot = 0
    for call in range(5):
        keys, off = requests(rng, pool, R, lo, hi)
        N = keys.shape[0]
        slots = np.arange(slot, slot + N, dtype=np.uint32)
        slot += N
        kd, od = to_dev(keys, torch.uint8), to_dev(off, torch.int64)
        hit, lslots = kt.lookup(kd, od)
        res, so = kt.store(kd, to_dev(slots), od, hit)
        whit, wslots = O.lookup(dt, keys, off)
        wres, wso = O.store_misses(dt, keys, off, whit, slots)
        kt.take_status()
        where = f"log2 {log2} R {R} call {call}"
        assert np.array_equal(hit.cpu().numpy(), whit), where
        assert np.array_equal(u32(lslots), wslots), where
        assert np.array_equal(res.cpu().numpy(), wres), where
        assert np.array_equal(u32(so), wso), where
        assert kt.entries() == len(dt)
        check_table(kt.table, dt, where)
    kt.close()


@pytest.mark.parametrize("log2", [3, 4, 6, 8, 10, 12])
@pytest.mark.parametrize("shape", SHAPES)
def test_lookup_store_crossing_capacity(log2, shape):
    R, lo, hi = shape
    cap = 1 << log2
    rng = np.random.default_rng(log2 * 17 + R)
    pool = pool_keys(rng, 2 * cap + 40)
    kt = KT(log2)
    dt = O.DictTable(cap)
    slot = 0
    for call in range(5):
        keys, off = requests(rng, pool, R, lo, hi)
        N = keys.shape[0]
        slots = np.arange(slot, slot + N, dtype=np.uint32)
        slot += N
        if call % 2:
            keys, slots = sprinkle(rng, keys, slots)
        hit, lslots, res, so = kt.lookup_store(to_dev(keys, torch.uint8), to_dev(off, torch.int64), to_dev(slots))
        whit, wslots = O.lookup(dt, keys, off)
        wres, wso = O.store_misses(dt, keys, off, whit, slots)
        kt.take_status()
        where = f"log2 {log2} R {R} call {call}"
        assert np.array_equal(hit.cpu().numpy(), whit), where
        assert np.array_equal(u32(lslots), wslots), where
        assert np.array_equal(res.cpu().numpy(), wres), where
        assert np.array_equal(u32(so), wso), where
        assert kt.entries() == len(dt)
        check_table(kt.table, dt, where)
    kt.close()


def test_lookup_store_work_taking_warps_crossing_capacity():
    """More requests than resident warps (the work-taking kernel) on a table
    of 2^12 entries that the batch overfills."""
    log2 = 12
    cap = 1 << log2
    rng = np.random.default_rng(99)
    pool = pool_keys(rng, 3 * cap)
    kt = KT(log2)
    dt = O.DictTable(cap)
    slot = 0
    for call in range(3):
        keys, off = requests(rng, pool, 40_000, 0, 3, dup_frac=0.5)
        N = keys.shape[0]
        slots = np.arange(slot, slot + N, dtype=np.uint32)
        slot += N
        hit, lslots, res, so = kt.lookup_store(to_dev(keys, torch.uint8), to_dev(off, torch.int64), to_dev(slots))
        whit, wslots = O.lookup(dt, keys, off)
        wres, wso = O.store_misses(dt, keys, off, whit, slots)
        kt.take_status()
        assert np.array_equal(hit.cpu().numpy(), whit)
        assert np.array_equal(u32(lslots), wslots)
        assert np.array_equal(res.cpu().numpy(), wres)
        assert np.array_equal(u32(so), wso)
        check_table(kt.table, dt, f"call {call}")
    kt.close()


@pytest.mark.parametrize("log2", [4, 7, 10, 12])
def test_derive_lookup_store_crossing_capacity(log2):
    """The whole hot path in one call on a table the batch overfills."""
    wl = W.reduced("small_block")
    C = wl.chunk_tokens
    cap = 1 << log2
    kt = KT(log2, C=C)
    dt = O.DictTable(cap)
    b = wl.batch
    d = O.descriptor_digests(wl.descriptors)
    rko, rkeys = O.derive_keys(b.tokens, b.tok_off, C, b.desc_idx, d)
    assert rkeys.shape[0] >= cap  # the batch alone overfills the table
    for call in range(2):
        nslots = np.arange(b.n_tokens // C, dtype=np.uint32) + 7 * call
        dg, key_off, keys, hit, lslots, res, so = kt.derive_lookup_store(b.tokens, b.tok_off, b.desc_idx,
                                                                        wl.descriptors, nslots)
        N = rkeys.shape[0]
        whit, wslots = O.lookup(dt, rkeys, rko)
        wres, wso = O.store_misses(dt, rkeys, rko, whit, nslots[:N])
        kt.take_status()
        assert np.array_equal(key_off.cpu().numpy(), rko)
        assert np.array_equal(keys.cpu().numpy()[:N], rkeys)
        assert np.array_equal(hit.cpu().numpy(), whit)
        assert np.array_equal(u32(lslots)[:N], wslots)
        assert np.array_equal(res.cpu().numpy()[:N], wres)
        assert np.array_equal(u32(so)[:N], wso)
        check_table(kt.table, dt, f"call {call}")
    kt.close()


# ---------------------------------------------------------------------------
# budget mode: stamps of refused keys
# ---------------------------------------------------------------------------
def triples(kt):
    e = kt.table.view(-1, 32).cpu().numpy()
    st = kt.stamps.cpu().numpy().view(np.uint64)
    occ = e[:, :16].any(axis=1)
    slots = e[:, 16:20].copy().view(np.uint32)[:, 0]
    assert not st[~occ].any(), "an empty entry holds a stamp"
    return sorted(zip((bytes(k) for k in e[occ, :16]), slots[occ].tolist(), st[occ].tolist()))


@pytest.mark.parametrize("log2", [5, 9])
def test_budget_mode_crossing_capacity(log2):
    cap = 1 << log2
    rng = np.random.default_rng(50 + log2)
    pool = pool_keys(rng, 2 * cap)
    kt = KT(log2)
    kt.attach_stamps()
    bt = O.BudgetTable(cap)
    slot = 0
    for call in range(6):
        if call % 2 == 0:
            keys = draw(rng, pool, cap // 2, 0.3)
            slots = np.arange(slot, slot + keys.shape[0], dtype=np.uint32)
            res, so = kt.store(to_dev(keys, torch.uint8), to_dev(slots))
            wres, wso = bt.store(keys, slots)
        else:
            keys, off = requests(rng, pool, 30, 1, 12)
            slots = np.arange(slot, slot + keys.shape[0], dtype=np.uint32)
            _, _, res, so = kt.lookup_store(to_dev(keys, torch.uint8), to_dev(off, torch.int64), to_dev(slots))
            _, _, wres, wso = bt.lookup_store(keys, off, slots)
        slot += keys.shape[0]
        kt.take_status()
        assert np.array_equal(res.cpu().numpy(), wres), f"call {call}"
        assert np.array_equal(u32(so), wso), f"call {call}"
        assert triples(kt) == bt.triples(), f"call {call}: stamps"
        assert empty_entries(kt.table) >= 1
    kt.close()


# ---------------------------------------------------------------------------
# the allocation-free store
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("log2", [3, 6, 9, 12])
def test_noalloc_crossing_capacity(log2):
    cap = 1 << log2
    rng = np.random.default_rng(200 + log2)
    pool = pool_keys(rng, 2 * cap + 5)
    table = torch.zeros(pk.pk_table_bytes(log2), dtype=torch.uint8, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    dt = O.DictTable(cap)
    slot = 0
    for call in range(6):
        if call % 2 == 0:
            n = int(rng.integers(max(1, cap // 4), 2 * cap + 1))
            keys = draw(rng, pool, n, 0.4)
            slots = np.arange(slot, slot + n, dtype=np.uint32)
            kd = to_dev(keys, torch.uint8)
            res = torch.empty(n, dtype=torch.int32, device="cuda")
            so = torch.empty_like(res)
            pk.pk_store_noalloc(table, log2, kd, to_dev(slots), res, so, status)
            wres, wso = dt.store(keys, slots)
        else:
            # range mode: the miss ranges of a lookup against the oracle's table
            keys, off = requests(rng, pool, 25, 1, 10)
            n = keys.shape[0]
            slots = np.arange(slot, slot + n, dtype=np.uint32)
            whit, _ = O.lookup(dt, keys, off)
            res = torch.empty(n, dtype=torch.int32, device="cuda")
            so = torch.empty_like(res)
            pk.pk_store_noalloc(table, log2, to_dev(keys, torch.uint8), to_dev(slots), res, so, status,
                                key_off=to_dev(off, torch.int64), hit_chunks=to_dev(whit))
            wres, wso = O.store_misses(dt, keys, off, whit, slots)
        slot += n
        torch.cuda.synchronize()
        status.zero_()
        assert np.array_equal(res.cpu().numpy(), wres), f"log2 {log2} call {call}"
        assert np.array_equal(u32(so), wso), f"log2 {log2} call {call}"
        check_table(table, dt, f"log2 {log2} call {call}")
