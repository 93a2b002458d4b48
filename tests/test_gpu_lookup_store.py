"""GPU parity of pk_lookup_store, the lookup and the store of the misses in one
pass, against the oracle's lookup followed by store_misses, and against the
two separate entry points on identical tables.  Bit-exact on every hit
length, slot, store result and output slot; tables compared as (key, slot)
sets, since which empty entry a racing insertion takes is not specified."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_38706_gb300 import workloads as W

pytestmark = pytest.mark.gpu

REDUCED = ["tiny", "multi_adapter", "small_block", "long_context", "provenance_sweep_D1",
           "provenance_sweep_D4", "provenance_sweep_D16", "provenance_sweep_D64"]
FULL = ["multi_adapter", "small_block", "long_context", "provenance_sweep_D1", "provenance_sweep_D4",
        "provenance_sweep_D16", "provenance_sweep_D64"]


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def _pairs(table: torch.Tensor):
    e = table.view(-1, 32).cpu().numpy()
    occ = e[:, :16].any(axis=1)
    slots = e[:, 16:20].copy().view(np.uint32)[:, 0]
    return sorted(zip((bytes(k) for k in e[occ, :16]), slots[occ].tolist()))


def seeded(wl):
    from paper_2609_38706_gb300.service import KeyTable
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    d = kt.digests(wl.descriptors)
    pko, pkeys = kt.derive(wl.prior.tokens, wl.prior.tok_off, wl.prior.desc_idx, d)
    pko_h = pko.cpu().numpy()
    kt.seed(W.seed_list(pkeys.cpu().numpy()[: int(pko_h[-1])], pko_h, wl.prior_chunks), wl.filler,
            wl.target_entries)
    assert kt.entries() == wl.target_entries
    return kt, d


def oracle_step(wl, keys, ko, new_slots, table_cls):
    d = O.descriptor_digests(wl.descriptors)
    pko, pk = O.derive_keys(wl.prior.tokens, wl.prior.tok_off, wl.chunk_tokens, wl.prior.desc_idx, d)
    t = O.seed_table(table_cls(wl.capacity), W.seed_list(pk, pko, wl.prior_chunks), wl.filler, wl.target_entries)
    hit, slots = O.lookup(t, keys, ko)
    res, so = O.store_misses(t, keys, ko, hit, new_slots)
    hit2, slots2 = O.lookup(t, keys, ko)
    return hit, slots, res, so, hit2, slots2, len(t)


def fused_vs_oracle(wl, table_cls, store_base=10_000_000):
    from paper_2609_38706_gb300.service import u32
    kt, d = seeded(wl)
    b = wl.batch
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
    kt.check("derive")
    N = int(key_off[-1])
    new_slots = np.arange(keys.shape[0], dtype=np.uint32) + store_base
    hit, slots, res, so = kt.lookup_store(keys, key_off, new_slots)
    kt.check("lookup_store")
    hit2, slots2 = kt.lookup(keys, key_off)
    kt.check("lookup after")
    ko = key_off.cpu().numpy()
    kh = keys.cpu().numpy()[:N]
    r = oracle_step(wl, kh, ko, new_slots[:N], table_cls)
    assert np.array_equal(hit.cpu().numpy(), r[0]), "hit lengths"
    assert np.array_equal(u32(slots)[:N], r[1]), "lookup slots"
    assert np.array_equal(res.cpu().numpy()[:N], r[2]), "store results"
    assert np.array_equal(u32(so)[:N], r[3]), "store slots"
    assert np.array_equal(hit2.cpu().numpy(), r[4]), "hit lengths after the call"
    assert np.array_equal(u32(slots2)[:N], r[5]), "slots after the call"
    assert kt.entries() == r[6]
    if wl.expected_hits is not None:
        assert np.array_equal(hit.cpu().numpy(), wl.expected_hits)
    kt.close()


@pytest.mark.parametrize("name", REDUCED)
def test_reduced_configs_bit_exact(name):
    fused_vs_oracle(W.reduced(name), O.DictTable)


@pytest.mark.slow
@pytest.mark.parametrize("name", FULL)
def test_full_configs_bit_exact(name):
    fused_vs_oracle(W.FULL_CONFIGS[name](), O.SortedTable)


@pytest.mark.parametrize("name", ["multi_adapter", "small_block", "long_context"])
def test_equals_separate_lookup_and_store(name):
    """Same table, same batch: pk_lookup_store == pk_lookup then pk_store."""
    wl = W.reduced(name)
    kt_a, d = seeded(wl)
    kt_b, _ = seeded(wl)
    b = wl.batch
    key_off, keys = kt_a.derive(b.tokens, b.tok_off, b.desc_idx, d)
    new_slots = torch.arange(keys.shape[0], dtype=torch.int32, device="cuda") + 777
    for call in range(2):  # the second call finds every key stored by the first
        hit_a, slots_a = kt_a.lookup(keys, key_off)
        res_a, so_a = kt_a.store(keys, new_slots, key_off, hit_a)
        hit_b, slots_b, res_b, so_b = kt_b.lookup_store(keys, key_off, new_slots)
        kt_a.check("separate")
        kt_b.check("fused")
        N = int(key_off[-1])
        assert torch.equal(hit_a, hit_b), f"call {call}: hit lengths"
        assert torch.equal(slots_a[:N], slots_b[:N]), f"call {call}: lookup slots"
        assert torch.equal(res_a, res_b), f"call {call}: results"
        assert torch.equal(so_a, so_b), f"call {call}: store slots"
        new_slots += 100_000
    assert kt_a.entries() == kt_b.entries()
    assert _pairs(kt_a.table) == _pairs(kt_b.table)
    kt_a.close()
    kt_b.close()


def _rows(rng, R, C, lo, hi):
    return [rng.integers(0, 50_000, int(rng.integers(lo, hi)) * C, dtype=np.int64).astype(np.int32)
            for _ in range(R)]


@pytest.mark.parametrize("shape", ["many_short", "few_long", "more_requests_than_warps"])
def test_reserved_slots_zero_keys_and_empty_requests(shape):
    """Keys whose new slot is PK_NO_SLOT (in the hit prefix: skipped; in the
    miss range: PK_ERR_ARG), all-zero keys, empty requests, duplicates across
    requests; the per-request path (many short requests), the per-key path
    (few long requests), and the per-request path with more requests than
    resident warps (warps take requests as they finish: 30,000 requests
    against 152 SMs x 3 CTAs x 8 warps on GB300)."""
    from paper_2609_38706_gb300.service import KeyTable, u32
    rng = np.random.default_rng({"many_short": 7, "few_long": 8, "more_requests_than_warps": 9}[shape])
    C = 16
    R, lo, hi = {"many_short": (1500, 0, 6), "few_long": (3, 200, 400),
                 "more_requests_than_warps": (30_000, 0, 6)}[shape]
    rows = _rows(rng, R, C, lo, hi)
    for r in range(1, R, 3):  # shared prefixes: duplicate keys across requests
        n = min(len(rows[r]), len(rows[r - 1]))
        rows[r][: n // 2] = rows[r - 1][: n // 2]
    toks = np.concatenate(rows)
    off = np.zeros(R + 1, np.int64)
    np.cumsum([len(x) for x in rows], out=off[1:])
    desc = [{"model_id": "m", "weight_precision": "bf16", "weight_version": "v", "adapter_id": "",
             "kv_format": "fp8_e4m3", "salt": ""}]
    didx = np.zeros(R, np.uint32)
    dd = O.descriptor_digests(desc)
    ko, keys = O.derive_keys(toks, off, C, didx, dd)
    N = keys.shape[0]
    keys = keys.copy()
    zero_at = rng.choice(N, size=max(1, N // 200), replace=False)
    keys[zero_at] = 0
    # seed: the first halves of every other request, so hit prefixes exist
    seed_idx = np.concatenate([np.arange(ko[r], ko[r] + (ko[r + 1] - ko[r]) // 2) for r in range(0, R, 2)])
    seed_idx = seed_idx[~np.isin(seed_idx, zero_at)]
    new_slots = np.arange(N, dtype=np.uint32) + 5000
    new_slots[rng.choice(N, size=max(1, N // 50), replace=False)] = O.NO_SLOT
    log2 = 14 if shape != "more_requests_than_warps" else 17
    t = O.DictTable(1 << log2)
    t.store(keys[seed_idx], seed_idx.astype(np.uint32))
    hit, slots = O.lookup(t, keys, ko)
    res, so = O.store_misses(t, keys, ko, hit, new_slots)

    kt = KeyTable(C, log2)
    kt.store(torch.from_numpy(keys[seed_idx]).cuda(), seed_idx.astype(np.uint32))
    kt.check("seed")
    g_hit, g_slots, g_res, g_so = kt.lookup_store(torch.from_numpy(keys).cuda(), torch.from_numpy(ko).cuda(),
                                                  new_slots)
    st = kt.take_status()
    assert np.array_equal(g_hit.cpu().numpy(), hit)
    assert np.array_equal(u32(g_slots), slots)
    assert np.array_equal(g_res.cpu().numpy(), res)
    assert np.array_equal(u32(g_so), so)
    errors = set(res[res < 0].tolist())
    assert (st != 0) == bool(errors) and (st == 0 or st in errors)
    assert O.PK_ERR_ARG in errors and O.PK_ERR_RESERVED_KEY in errors
    assert kt.entries() == len(t)
    kt.close()


def test_empty_batch():
    from paper_2609_38706_gb300.service import KeyTable
    kt = KeyTable(16, 6)
    keys = torch.zeros((0, 32), dtype=torch.uint8, device="cuda")
    key_off = torch.zeros(4, dtype=torch.int64, device="cuda")
    hit, slots, res, so = kt.lookup_store(keys, key_off, np.zeros(0, np.uint32))
    kt.check()
    assert hit.cpu().tolist() == [0, 0, 0]
    assert kt.entries() == 0
    kt.close()


@pytest.mark.parametrize("name", ["long_context", "multi_adapter"])
def test_store_reads_the_lookup_it_follows(name):
    """pk_lookup then pk_store in range mode as the last two calls, with the
    h_r buffer pre-filled with zeros: the store must act on the lookup's h_r
    (its kernels start while the lookup's are still running)."""
    from paper_2609_38706_gb300 import pk
    wl = W.reduced(name)
    kt, d = seeded(wl)
    b = wl.batch
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
    snap = kt.save()
    N = keys.shape[0]
    new_slots = torch.arange(N, dtype=torch.int32, device="cuda") + 777
    ko = key_off.cpu().numpy()
    r = oracle_step(wl, keys.cpu().numpy()[: int(ko[-1])], ko, new_slots.cpu().numpy()[: int(ko[-1])].astype(np.uint32),
                    O.DictTable)
    for _ in range(4):
        kt.load(snap)
        hit = torch.zeros(key_off.numel() - 1, dtype=torch.int32, device="cuda")
        slots = torch.empty(N, dtype=torch.int32, device="cuda")
        res = torch.full((N,), -55, dtype=torch.int32, device="cuda")
        so = torch.empty(N, dtype=torch.int32, device="cuda")
        torch.cuda.synchronize()
        pk.pk_lookup(kt.ctx, keys, key_off, hit, slots, kt.status, kt.stream)
        pk.pk_store(kt.ctx, keys, new_slots, res, so, kt.status, key_off, hit, kt.stream)
        torch.cuda.synchronize()
        kt.check("lookup, store")
        assert np.array_equal(hit.cpu().numpy(), r[0])
        assert np.array_equal(res.cpu().numpy()[: int(ko[-1])], r[2])
    kt.close()
