"""GPU test of pk_store_noalloc, the store entry point that allocates nothing.

Callers that cannot allocate device memory (engines whose device memory
belongs to their own fixed pool, latency-critical paths that must stay out of
the CUDA allocator) cannot create a libpk context, because pk_init
allocates the context's entry counter.  pk_store_noalloc serves them: it keeps
its scratch in a fixed device array inside the library.  Its results must be
those of pk_store (the context entry point) on the same inputs, call after
call.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def _pairs(table: torch.Tensor):
    """Stored (16-byte key, slot) pairs of a raw table, position-independent."""
    e = table.view(-1, 32).cpu().numpy()
    occ = e[:, :16].any(axis=1)
    slots = e[:, 16:20].copy().view(np.uint32)[:, 0]
    return sorted(zip((bytes(k) for k in e[occ, :16]), slots[occ].tolist()))


def test_noalloc_store_matches_pk_store_on_consecutive_calls():
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300.service import KeyTable

    log2 = 12
    kt = KeyTable(16, log2)                                        # context entry point
    table_b = torch.zeros(pk.pk_table_bytes(log2), dtype=torch.uint8, device="cuda")  # caller-owned, zeroed
    status_b = torch.zeros(1, dtype=torch.int32, device="cuda")
    rng = np.random.default_rng(123)
    pool = rng.integers(0, 256, (600, 32), dtype=np.uint8)
    pool[:, 0] |= 1                                                # no all-zero (reserved) keys
    for call in range(2):
        idx = rng.integers(0, pool.shape[0], 3000)                 # many duplicates within and across calls
        keys = torch.from_numpy(pool[idx]).cuda()
        slots = torch.from_numpy(rng.integers(0, 2**31, 3000).astype(np.int32)).cuda()
        res_a, out_a = kt.store(keys, slots)
        res_b = torch.empty_like(res_a)
        out_b = torch.empty_like(out_a)
        pk.pk_store_noalloc(table_b, log2, keys, slots, res_b, out_b, status_b)
        torch.cuda.synchronize()
        kt.check("pk_store")
        assert int(status_b.item()) == 0
        assert torch.equal(res_a, res_b), f"call {call}: results differ"
        assert torch.equal(out_a, out_b), f"call {call}: slots differ"
    assert _pairs(kt.table) == _pairs(table_b)
    kt.close()


def test_noalloc_range_mode_matches_pk_store():
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300 import workloads as W
    from paper_2609_38706_gb300.service import KeyTable

    wl = W.reduced("multi_adapter")
    log2 = wl.capacity_log2
    kt = KeyTable(wl.chunk_tokens, log2)
    d = kt.digests(wl.descriptors)
    pko, pkeys = kt.derive(wl.prior.tokens, wl.prior.tok_off, wl.prior.desc_idx, d)
    seed = pkeys[: int(pko[-1])]
    seed_slots = torch.arange(seed.shape[0], dtype=torch.int32, device="cuda")
    kt.store(seed, seed_slots)
    table_b = torch.zeros(pk.pk_table_bytes(log2), dtype=torch.uint8, device="cuda")
    status_b = torch.zeros(1, dtype=torch.int32, device="cuda")
    rb = torch.empty(seed.shape[0], dtype=torch.int32, device="cuda")
    ob = torch.empty_like(rb)
    pk.pk_store_noalloc(table_b, log2, seed.contiguous(), seed_slots, rb, ob, status_b)

    b = wl.batch
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
    hit, _ = kt.lookup(keys, key_off)
    new_slots = torch.arange(keys.shape[0], dtype=torch.int32, device="cuda") + 5000
    for call in range(2):
        res_a, out_a = kt.store(keys, new_slots, key_off, hit)
        res_b = torch.empty_like(res_a)
        out_b = torch.empty_like(out_a)
        pk.pk_store_noalloc(table_b, log2, keys, new_slots, res_b, out_b, status_b, key_off=key_off, hit_chunks=hit)
        torch.cuda.synchronize()
        kt.check("pk_store")
        assert int(status_b.item()) == 0
        assert torch.equal(res_a, res_b), f"call {call}: results differ"
        assert torch.equal(out_a, out_b), f"call {call}: slots differ"
    assert _pairs(kt.table) == _pairs(table_b)
    kt.close()


def test_noalloc_rejects_more_entries_than_its_scratch():
    from paper_2609_38706_gb300 import pk

    L = pk.lib()
    table = torch.zeros(pk.pk_table_bytes(6), dtype=torch.uint8, device="cuda")
    cfg = pk.pk_config(1, 6, 0, table.data_ptr(), table.numel())
    n = pk.PK_NOALLOC_MAX_ENTRIES + 1
    # rejected on the host before any pointer is used or anything is enqueued
    rc = L.pk_store_noalloc(ctypes.byref(cfg), None, None, n, None, None, 0, None, None, None, None)
    assert rc == pk.PK_ERR_TOO_LARGE
    assert "PK_NOALLOC_MAX_ENTRIES" in pk.pk_strerror(rc)
