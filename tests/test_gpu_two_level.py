"""GPU parity of the two-level variant: digests from the library's host
entry points (pk_worker_digest, pk_request_digest) folded into the device key
derivation, against the oracle's two-level digests and keys, bit-exact; the
inert requests (no adapter, no salt) key exactly as the worker-only chain."""
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


@pytest.mark.parametrize("name", ["tiny", "multi_adapter", "long_context", "provenance_sweep_D16"])
def test_two_level_keys_bit_exact(name):
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300.service import KeyTable
    wl = W.reduced(name)
    b = wl.batch
    dg = pk.two_level_digests(wl.descriptors)
    assert np.array_equal(dg, O.two_level_digests(wl.descriptors))
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, torch.from_numpy(dg).cuda())
    kt.check("derive")
    rko, rkeys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, O.two_level_digests(wl.descriptors))
    assert np.array_equal(key_off.cpu().numpy(), rko)
    got = keys.cpu().numpy()[: rkeys.shape[0]]
    assert np.array_equal(got, rkeys)
    # inert requests: the same keys as a derivation with the worker digest alone
    inert = [j for j, d in enumerate(wl.descriptors) if not d.get("adapter_id") and not d.get("salt")
             and not d.get("extra")]
    for j in inert:
        wdig = np.frombuffer(pk.pk_worker_digest(wl.descriptors[j]), np.uint8)
        assert np.array_equal(dg[j], wdig)
    kt.close()


def test_two_level_lookup_and_store_through_the_table():
    """Keys of the two-level variant go through the same table path: lookup and
    store of a batch, then a second lookup finds every key (oracle as reference)."""
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300.service import KeyTable, u32
    wl = W.reduced("multi_adapter")
    b = wl.batch
    dg = torch.from_numpy(pk.two_level_digests(wl.descriptors)).cuda()
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    pko, pkeys = kt.derive(wl.prior.tokens, wl.prior.tok_off, wl.prior.desc_idx, dg)
    pko_h = pko.cpu().numpy()
    seeds = W.seed_list(pkeys.cpu().numpy()[: int(pko_h[-1])], pko_h, wl.prior_chunks)
    kt.seed(seeds, wl.filler, wl.target_entries)
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, dg)
    N = int(key_off[-1])
    new_slots = np.arange(keys.shape[0], dtype=np.uint32) + 90_000
    hit, slots, res, so = kt.lookup_store(keys, key_off, new_slots)
    kt.check("lookup_store")
    rd = O.two_level_digests(wl.descriptors)
    rpko, rpk = O.derive_keys(wl.prior.tokens, wl.prior.tok_off, wl.chunk_tokens, wl.prior.desc_idx, rd)
    t = O.seed_table(O.DictTable(wl.capacity), W.seed_list(rpk, rpko, wl.prior_chunks), wl.filler,
                     wl.target_entries)
    rko, rkeys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, rd)
    rhit, rslots = O.lookup(t, rkeys, rko)
    rres, rso = O.store_misses(t, rkeys, rko, rhit, new_slots[:N])
    assert np.array_equal(hit.cpu().numpy(), rhit)
    assert np.array_equal(u32(slots)[:N], rslots)
    assert np.array_equal(res.cpu().numpy()[:N], rres)
    assert np.array_equal(u32(so)[:N], rso)
    kt.close()
