"""GPU parity: the CUDA path through the C-ABI against the CPU oracle.

Bit-exact on every descriptor digest, chunk offset, key, hit length, slot and
store result.  Reduced, ragged variants of every configuration run element by
element (many thread blocks, partial trailing chunks, unaligned request
starts, empty requests); the full-size configurations (marked slow) compare
every key and every probe result against the oracle's sort-based table.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_38706_gb300 import workloads as W

pytestmark = pytest.mark.gpu

REDUCED = ["tiny", "multi_adapter", "small_block", "long_context", "provenance_sweep_D1",
           "provenance_sweep_D4", "provenance_sweep_D16", "provenance_sweep_D64"]


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def run_gpu(wl, store_base=10_000_000):
    from paper_2609_38706_gb300.service import KeyTable, u32
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    out = {}
    d = kt.digests(wl.descriptors)
    out["digests"] = d.cpu().numpy()
    pko, pkeys = kt.derive(wl.prior.tokens, wl.prior.tok_off, wl.prior.desc_idx, d)
    pko_h = pko.cpu().numpy()
    pkeys_h = pkeys.cpu().numpy()[: int(pko_h[-1])]
    out["prior_keys"] = pkeys_h
    kt.seed(W.seed_list(pkeys_h, pko_h, wl.prior_chunks), wl.filler, wl.target_entries)
    out["entries_seeded"] = kt.entries()
    b = wl.batch
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
    kt.check("derive")
    N = int(key_off[-1])
    hit, slots = kt.lookup(keys, key_off)
    kt.check("lookup")
    new_slots = np.arange(keys.shape[0], dtype=np.uint32) + store_base
    res, so = kt.store(keys, new_slots, key_off, hit)
    kt.check("store")
    hit2, slots2 = kt.lookup(keys, key_off)
    kt.check("lookup2")
    out.update(key_off=key_off.cpu().numpy(), keys=keys.cpu().numpy()[:N], hit=hit.cpu().numpy(),
               slots=u32(slots)[:N], result=res.cpu().numpy()[:N], slot_out=u32(so)[:N],
               hit2=hit2.cpu().numpy(), slots2=u32(slots2)[:N], entries=kt.entries(), new_slots=new_slots)
    kt.close()
    return out


def run_oracle(wl, new_slots, table_cls):
    C = wl.chunk_tokens
    d = O.descriptor_digests(wl.descriptors)
    pko, pk = O.derive_keys(wl.prior.tokens, wl.prior.tok_off, C, wl.prior.desc_idx, d)
    t = O.seed_table(table_cls(wl.capacity), W.seed_list(pk, pko, wl.prior_chunks), wl.filler, wl.target_entries)
    seeded = len(t)
    b = wl.batch
    ko, keys = O.derive_keys(b.tokens, b.tok_off, C, b.desc_idx, d)
    hit, slots = O.lookup(t, keys, ko)
    res, so = O.store_misses(t, keys, ko, hit, new_slots[: keys.shape[0]])
    hit2, slots2 = O.lookup(t, keys, ko)
    return dict(digests=d, prior_keys=pk, entries_seeded=seeded, key_off=ko, keys=keys, hit=hit, slots=slots,
                result=res, slot_out=so, hit2=hit2, slots2=slots2, entries=len(t))


def compare(g, r, wl):
    assert np.array_equal(g["digests"], r["digests"]), "descriptor digests"
    assert np.array_equal(g["prior_keys"], r["prior_keys"]), "prior batch keys"
    assert g["entries_seeded"] == r["entries_seeded"] == wl.target_entries
    assert np.array_equal(g["key_off"], r["key_off"]), "key offsets"
    assert np.array_equal(g["keys"], r["keys"]), "keys"
    assert np.array_equal(g["hit"], r["hit"]), "hit lengths"
    assert np.array_equal(g["slots"], r["slots"]), "slots"
    assert np.array_equal(g["result"], r["result"]), "store results"
    assert np.array_equal(g["slot_out"], r["slot_out"]), "store slots"
    assert np.array_equal(g["hit2"], r["hit2"]), "hit lengths after store"
    assert np.array_equal(g["slots2"], r["slots2"]), "slots after store"
    assert g["entries"] == r["entries"]
    if wl.expected_hits is not None:
        assert np.array_equal(g["hit"], wl.expected_hits), "generator-known hit lengths"


@pytest.mark.parametrize("name", REDUCED)
def test_reduced_configs_bit_exact(name):
    wl = W.reduced(name)
    g = run_gpu(wl)
    r = run_oracle(wl, g["new_slots"], O.DictTable)
    compare(g, r, wl)
    assert np.array_equal(g["hit2"], np.diff(g["key_off"]))


FULL = ["multi_adapter", "small_block", "long_context", "provenance_sweep_D1", "provenance_sweep_D4",
        "provenance_sweep_D16", "provenance_sweep_D64"]


@pytest.mark.slow
@pytest.mark.parametrize("name", FULL)
def test_full_configs_every_key(name):
    wl = W.FULL_CONFIGS[name]()
    g = run_gpu(wl)
    r = run_oracle(wl, g["new_slots"], O.SortedTable)
    compare(g, r, wl)
    if name.startswith("provenance_sweep"):
        D = wl.notes["D"]
        assert len({bytes(x) for x in O.prefix128(g["prior_keys"])}) == 16 * D   # Sec. 6.5 storage growth


@pytest.mark.parametrize("name", REDUCED)
def test_fused_descriptor_and_key_derivation(name):
    """pk_derive_keys_enc: digests d and keys from one launch sequence."""
    from paper_2609_38706_gb300.service import KeyTable
    wl = W.reduced(name)
    b = wl.batch
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    d, ko, keys = kt.derive_enc(b.tokens, b.tok_off, b.desc_idx, wl.descriptors)
    kt.check("derive_enc")
    rd = O.descriptor_digests(wl.descriptors)
    rko, rkeys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, rd)
    assert np.array_equal(d.cpu().numpy(), rd)
    assert np.array_equal(ko.cpu().numpy(), rko)
    assert np.array_equal(keys.cpu().numpy()[: rkeys.shape[0]], rkeys)
    kt.close()


def test_fused_empty_batch():
    from paper_2609_38706_gb300.service import KeyTable
    kt = KeyTable(16, 6)
    d, ko, keys = kt.derive_enc(np.zeros(0, np.int32), np.zeros(1, np.int64), np.zeros(0, np.uint32),
                                [W.tiny().descriptors[0]])
    kt.check()
    assert ko.cpu().tolist() == [0] and keys.shape[0] == 0
    assert d.cpu().numpy().tobytes() == O.descriptor_digest(W.tiny().descriptors[0])
    kt.close()


def test_cross_context_stability():
    """Two independent contexts (two 'workers') derive identical keys."""
    from paper_2609_38706_gb300.service import KeyTable
    wl = W.reduced("multi_adapter")
    b = wl.batch
    outs = []
    for _ in range(2):
        kt = KeyTable(wl.chunk_tokens, 10)
        d = kt.digests(wl.descriptors)
        ko, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
        outs.append(keys.cpu().numpy()[: int(ko[-1])])
        kt.close()
    assert np.array_equal(outs[0], outs[1])


def test_side_stream():
    from paper_2609_38706_gb300.service import KeyTable
    wl = W.tiny()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        kt = KeyTable(wl.chunk_tokens, wl.capacity_log2, stream=s)
        d = kt.digests(wl.descriptors)
        ko, keys = kt.derive(wl.batch.tokens, wl.batch.tok_off, wl.batch.desc_idx, d)
    s.synchronize()
    rko, rkeys = O.derive_keys(wl.batch.tokens, wl.batch.tok_off, wl.chunk_tokens, wl.batch.desc_idx,
                               O.descriptor_digests(wl.descriptors))
    assert np.array_equal(keys.cpu().numpy(), rkeys)
    kt.close()
