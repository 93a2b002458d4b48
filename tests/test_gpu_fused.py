"""GPU parity of pk_derive_lookup_store, the whole hot path in one call,
against the oracle's key derivation, lookup and store of the misses, and
against pk_derive_keys_enc followed by pk_lookup_store on identical tables.
Bit-exact on every key, hit length, lookup slot, store result and output
slot; tables compared as (key, slot) sets."""
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


def seeded(wl, stamps=False):
    from paper_2609_38706_gb300.service import KeyTable
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    if stamps:
        kt.attach_stamps()
    d = kt.digests(wl.descriptors)
    pko, pkeys = kt.derive(wl.prior.tokens, wl.prior.tok_off, wl.prior.desc_idx, d)
    pko_h = pko.cpu().numpy()
    seeds = W.seed_list(pkeys.cpu().numpy()[: int(pko_h[-1])], pko_h, wl.prior_chunks)
    kt.seed(seeds, wl.filler, wl.target_entries)
    return kt, seeds


def check_vs_oracle(wl, table_cls):
    from paper_2609_38706_gb300.service import u32
    kt, _ = seeded(wl)
    b = wl.batch
    cap = b.n_tokens // wl.chunk_tokens
    new_slots = np.arange(cap, dtype=np.uint32) + 10_000_000
    dg, key_off, keys, hit, slots, res, so = kt.derive_lookup_store(b.tokens, b.tok_off, b.desc_idx, wl.descriptors,
                                                                    new_slots)
    kt.check("derive_lookup_store")
    ko = key_off.cpu().numpy()
    N = int(ko[-1])
    d = O.descriptor_digests(wl.descriptors)
    oko, okeys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d)
    assert np.array_equal(dg.cpu().numpy(), d)
    assert np.array_equal(ko, oko)
    assert np.array_equal(keys.cpu().numpy()[:N], okeys)
    pko, pk_ = O.derive_keys(wl.prior.tokens, wl.prior.tok_off, wl.chunk_tokens, wl.prior.desc_idx, d)
    t = O.seed_table(table_cls(wl.capacity), W.seed_list(pk_, pko, wl.prior_chunks), wl.filler, wl.target_entries)
    oh, osl = O.lookup(t, okeys, oko)
    ores, oso = O.store_misses(t, okeys, oko, oh, new_slots[:N])
    assert np.array_equal(hit.cpu().numpy(), oh), "hit lengths"
    assert np.array_equal(u32(slots)[:N], osl), "lookup slots"
    assert np.array_equal(res.cpu().numpy()[:N], ores), "store results"
    assert np.array_equal(u32(so)[:N], oso), "store slots"
    assert kt.entries() == len(t)
    if wl.expected_hits is not None:
        assert np.array_equal(hit.cpu().numpy(), wl.expected_hits)
    kt.close()


@pytest.mark.parametrize("name", REDUCED)
def test_reduced_configs_bit_exact(name):
    check_vs_oracle(W.reduced(name), O.DictTable)


@pytest.mark.slow
@pytest.mark.parametrize("name", FULL)
def test_full_configs_bit_exact(name):
    check_vs_oracle(W.FULL_CONFIGS[name](), O.SortedTable)


@pytest.mark.parametrize("name", ["multi_adapter", "small_block", "long_context"])
def test_equals_the_two_calls(name):
    """Same table, same batch: pk_derive_lookup_store == pk_derive_keys_enc then
    pk_lookup_store, call after call (the second finds every key stored)."""
    wl = W.reduced(name)
    kt_a, _ = seeded(wl)
    kt_b, _ = seeded(wl)
    b = wl.batch
    cap = b.n_tokens // wl.chunk_tokens
    new_slots = np.arange(cap, dtype=np.uint32) + 777
    new_slots[::7] = O.NO_SLOT  # some keys only looked up
    for call in range(2):
        _, ko_a, keys_a = kt_a.derive_enc(b.tokens, b.tok_off, b.desc_idx, wl.descriptors)
        ha, sa, ra, oa = kt_a.lookup_store(keys_a, ko_a, new_slots)
        _, ko_b, keys_b, hb, sb, rb, ob = kt_b.derive_lookup_store(b.tokens, b.tok_off, b.desc_idx, wl.descriptors,
                                                                   new_slots)
        sta, stb = kt_a.take_status(), kt_b.take_status()
        assert sta == stb
        N = int(ko_a[-1])
        assert torch.equal(ko_a, ko_b) and torch.equal(keys_a[:N], keys_b[:N])
        assert torch.equal(ha, hb), f"call {call}: hit lengths"
        assert torch.equal(sa[:N], sb[:N]), f"call {call}: lookup slots"
        assert torch.equal(ra[:N], rb[:N]), f"call {call}: results"
        assert torch.equal(oa[:N], ob[:N]), f"call {call}: store slots"
        new_slots = new_slots + 100_000
        new_slots[::7] = O.NO_SLOT
    assert kt_a.entries() == kt_b.entries()
    assert _pairs(kt_a.table) == _pairs(kt_b.table)
    kt_a.close()
    kt_b.close()


def test_budget_mode_stamps():
    """Stamps raised by the fused call equal the oracle's budget table."""
    wl = W.reduced("multi_adapter")
    kt, seeds = seeded(wl, stamps=True)
    bt = O.BudgetTable(wl.capacity)
    if seeds.shape[0]:
        bt.store(seeds, np.arange(seeds.shape[0], dtype=np.uint32))
    need = wl.target_entries - len(bt)
    if need > 0:
        bt.store(wl.filler[:need], np.arange(seeds.shape[0], seeds.shape[0] + need, dtype=np.uint32))
    b = wl.batch
    cap = b.n_tokens // wl.chunk_tokens
    new_slots = np.arange(cap, dtype=np.uint32) + 5_000_000
    _, key_off, keys, hit, _, _, _ = kt.derive_lookup_store(b.tokens, b.tok_off, b.desc_idx, wl.descriptors, new_slots)
    kt.check()
    N = int(key_off[-1])
    bt.lookup_store(keys.cpu().numpy()[:N], key_off.cpu().numpy(), new_slots[:N])
    e = kt.table.view(-1, 32).cpu().numpy()
    st = kt.stamps.cpu().numpy().view(np.uint64)
    occ = e[:, :16].any(axis=1)
    slots = e[:, 16:20].copy().view(np.uint32)[:, 0]
    got = sorted(zip((bytes(k) for k in e[occ, :16]), slots[occ].tolist(), st[occ].tolist()))
    assert got == bt.triples()
    kt.close()


def test_budget_mode_stamps_with_more_requests_than_warps():
    """Stamps raised by pk_lookup_store when its warps take requests from a
    counter (30,000 short requests against 152 SMs x 3 CTAs x 8 warps on
    GB300): which warp serves a request must not change any stamp, slot or
    result, so they equal the oracle's budget table."""
    from paper_2609_38706_gb300.service import KeyTable, u32
    rng = np.random.default_rng(31)
    C, R = 16, 30_000
    rows = [rng.integers(0, 40_000, int(rng.integers(0, 6)) * C, dtype=np.int64).astype(np.int32) for _ in range(R)]
    for r in range(1, R, 3):  # shared prefixes: the same keys in several requests
        n = min(len(rows[r]), len(rows[r - 1]))
        rows[r][: n // 2] = rows[r - 1][: n // 2]
    toks = np.concatenate(rows)
    off = np.zeros(R + 1, np.int64)
    np.cumsum([len(x) for x in rows], out=off[1:])
    desc = [{"model_id": "m", "weight_precision": "bf16", "weight_version": "v", "adapter_id": "",
             "kv_format": "bf16", "salt": ""}]
    ko, keys = O.derive_keys(toks, off, C, np.zeros(R, np.uint32), O.descriptor_digests(desc))
    N = keys.shape[0]
    seed_idx = np.concatenate([np.arange(ko[r], ko[r] + (ko[r + 1] - ko[r]) // 2) for r in range(0, R, 2)])
    log2 = 17
    kt = KeyTable(C, log2)
    kt.attach_stamps()
    kt.store(torch.from_numpy(keys[seed_idx]).cuda(), seed_idx.astype(np.uint32))
    kt.check("seed")
    bt = O.BudgetTable(1 << log2)
    bt.store(keys[seed_idx], seed_idx.astype(np.uint32))
    new_slots = np.arange(N, dtype=np.uint32) + 5_000_000
    hit, slots, res, so = kt.lookup_store(torch.from_numpy(keys).cuda(), torch.from_numpy(ko).cuda(), new_slots)
    kt.check("lookup_store")
    t = O.DictTable(1 << log2)
    t.store(keys[seed_idx], seed_idx.astype(np.uint32))
    r_hit, r_slots = O.lookup(t, keys, ko)
    r_res, r_so = O.store_misses(t, keys, ko, r_hit, new_slots)
    assert np.array_equal(hit.cpu().numpy(), r_hit)
    assert np.array_equal(u32(slots), r_slots)
    assert np.array_equal(res.cpu().numpy(), r_res)
    assert np.array_equal(u32(so), r_so)
    bt.lookup_store(keys, ko, new_slots)
    e = kt.table.view(-1, 32).cpu().numpy()
    st = kt.stamps.cpu().numpy().view(np.uint64)
    occ = e[:, :16].any(axis=1)
    tslots = e[:, 16:20].copy().view(np.uint32)[:, 0]
    got = sorted(zip((bytes(k) for k in e[occ, :16]), tslots[occ].tolist(), st[occ].tolist()))
    assert got == bt.triples()
    kt.close()


@pytest.mark.parametrize("shape", ["empty_batch", "no_full_chunks", "mixed"])
def test_empty_and_short_requests(shape):
    from paper_2609_38706_gb300.service import KeyTable, u32
    C = 16
    rng = np.random.default_rng(3)
    if shape == "empty_batch":
        lens = [0, 0, 0]
    elif shape == "no_full_chunks":
        lens = [5, 15, 0, 1]
    else:
        lens = [0, 33, 15, 16, 700, 0, 48] * 9
    rows = [rng.integers(0, 50_000, n, dtype=np.int64).astype(np.int32) for n in lens]
    toks = np.concatenate(rows) if sum(lens) else np.zeros(0, np.int32)
    off = np.zeros(len(lens) + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    desc = [{"model_id": "m", "weight_precision": "bf16", "weight_version": "v", "adapter_id": "", "kv_format": "bf16",
             "salt": ""}]
    didx = np.zeros(len(lens), np.uint32)
    kt = KeyTable(C, 12)
    cap = toks.size // C
    new_slots = np.arange(max(cap, 1), dtype=np.uint32)[:cap]
    _, key_off, keys, hit, slots, res, so = kt.derive_lookup_store(toks, off, didx, desc, new_slots)
    kt.check()
    d = O.descriptor_digests(desc)
    oko, okeys = O.derive_keys(toks, off, C, didx, d)
    t = O.DictTable(1 << 12)
    oh, osl = O.lookup(t, okeys, oko)
    ores, oso = O.store_misses(t, okeys, oko, oh, new_slots[: okeys.shape[0]])
    N = int(oko[-1])
    assert np.array_equal(key_off.cpu().numpy(), oko)
    assert np.array_equal(hit.cpu().numpy(), oh)
    assert np.array_equal(u32(slots)[:N], osl) and np.array_equal(res.cpu().numpy()[:N], ores)
    assert np.array_equal(u32(so)[:N], oso)
    assert kt.entries() == len(t)
    kt.close()


def test_host_argument_errors():
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300.service import KeyTable
    kt = KeyTable(16, 8)
    L = pk.lib()
    fake = 1 << 40
    # R > 0 without hit_chunks; key_capacity too small; misaligned outputs
    assert L.pk_derive_lookup_store(kt.ctx, fake, 64, fake, 2, fake, fake, 10, fake, 1, fake, fake, fake, 4, fake,
                                    None, fake, fake, fake, None, None) == pk.PK_ERR_ARG
    assert L.pk_derive_lookup_store(kt.ctx, fake, 64, fake, 2, fake, fake, 10, fake, 1, fake, fake, fake, 3, fake,
                                    fake, fake, fake, fake, None, None) == pk.PK_ERR_ARG
    assert L.pk_derive_lookup_store(kt.ctx, fake, 64, fake, 2, fake, fake, 10, fake, 1, fake, fake, fake, 4, fake,
                                    fake, fake + 2, fake, fake, None, None) == pk.PK_ERR_ARG
    kt.close()
