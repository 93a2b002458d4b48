"""GPU tests of checkpoint and resume (the shared store outlives workers,
Sec. 2.1): pk_table_save / pk_table_load through device memory (one-pass load
kernel) and through pinned host memory (copy, then the marking kernel).  A
loaded table must hold the saved keys and slots byte for byte, count its
entries, mark them as inserted before any later call (epoch 1, no claim
owner), answer lookups as the saved one did, and store the next batch as the
oracle does; attached stamps are zeroed."""
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


def _entries(table: torch.Tensor):
    e = table.view(-1, 32).cpu().numpy()
    occ = e[:, :16].any(axis=1)
    words = e.view(np.uint32)  # [cap, 8]: key (4), slot, owner, epoch lo, epoch hi
    return e, occ, words


def _seeded(wl):
    from paper_2609_38706_gb300.service import KeyTable
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    d = kt.digests(wl.descriptors)
    pko, pkeys = kt.derive(wl.prior.tokens, wl.prior.tok_off, wl.prior.desc_idx, d)
    pko_h = pko.cpu().numpy()
    kt.seed(W.seed_list(pkeys.cpu().numpy()[: int(pko_h[-1])], pko_h, wl.prior_chunks), wl.filler,
            wl.target_entries)
    return kt, d


@pytest.mark.parametrize("where", ["device", "host"])
@pytest.mark.parametrize("name", ["multi_adapter", "small_block"])
def test_save_load_into_a_new_context(where, name):
    from paper_2609_38706_gb300.service import KeyTable, u32
    wl = W.reduced(name)
    kt, d = _seeded(wl)
    b = wl.batch
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
    N = int(key_off[-1])
    nbytes = kt.table.numel() + 64
    dst = (torch.empty(nbytes, dtype=torch.uint8, device="cuda") if where == "device"
           else torch.empty(nbytes, dtype=torch.uint8).pin_memory())
    kt.save(dst)
    torch.cuda.synchronize()
    kt2 = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    kt2.load(dst)
    torch.cuda.synchronize()
    kt2.check("load")
    assert kt2.entries() == kt.entries() == wl.target_entries
    e1, occ1, w1 = _entries(kt.table)
    e2, occ2, w2 = _entries(kt2.table)
    assert np.array_equal(occ1, occ2)
    assert np.array_equal(e1[:, :20], e2[:, :20])           # keys and slots byte for byte
    assert (w2[occ2, 5] == 0).all()                          # no claim owner
    assert (w2[occ2, 6] == 1).all() and (w2[occ2, 7] == 0).all()  # epoch 1
    assert not e2[~occ2].any()                               # empty entries stay all zero
    h1, s1 = kt.lookup(keys, key_off)
    h2, s2 = kt2.lookup(keys, key_off)
    assert torch.equal(h1, h2) and torch.equal(s1[:N], s2[:N])
    # the next lookup-and-store on the loaded table equals the oracle's on the seeded one
    new_slots = np.arange(keys.shape[0], dtype=np.uint32) + 9_000_000
    hit, slots, res, so = kt2.lookup_store(keys, key_off, new_slots)
    kt2.check("lookup_store")
    ko = key_off.cpu().numpy()
    pko, pk_ = O.derive_keys(wl.prior.tokens, wl.prior.tok_off, wl.chunk_tokens, wl.prior.desc_idx,
                             O.descriptor_digests(wl.descriptors))
    t = O.seed_table(O.DictTable(wl.capacity), W.seed_list(pk_, pko, wl.prior_chunks), wl.filler, wl.target_entries)
    kh = keys.cpu().numpy()[:N]
    oh, osl = O.lookup(t, kh, ko)
    ores, oso = O.store_misses(t, kh, ko, oh, new_slots[:N])
    assert np.array_equal(hit.cpu().numpy(), oh)
    assert np.array_equal(u32(slots)[:N], osl)
    assert np.array_equal(res.cpu().numpy()[:N], ores)
    assert np.array_equal(u32(so)[:N], oso)
    assert kt2.entries() == len(t)
    kt.close()
    kt2.close()


def test_restore_into_the_same_context_repeats_the_step():
    wl = W.reduced("multi_adapter")
    kt, d = _seeded(wl)
    b = wl.batch
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
    snap = kt.save()
    N = int(key_off[-1])  # outputs past the batch's keys are not written
    new_slots = np.arange(keys.shape[0], dtype=np.uint32) + 1234
    outs = []
    for _ in range(3):
        kt.load(snap)
        hit, slots, res, so = kt.lookup_store(keys, key_off, new_slots)
        kt.check("step")
        outs.append((hit.cpu(), slots.cpu()[:N], res.cpu()[:N], so.cpu()[:N], kt.entries()))
    for o in outs[1:]:
        assert all(torch.equal(a, b_) for a, b_ in zip(o[:4], outs[0][:4])) and o[4] == outs[0][4]
    kt.close()


def test_load_zeroes_attached_stamps():
    from paper_2609_38706_gb300.service import KeyTable
    rng = np.random.default_rng(4)
    kt = KeyTable(16, 10)
    kt.attach_stamps()
    keys = rng.integers(0, 256, (300, 32), dtype=np.uint8)
    keys[:, 0] |= 1
    kt.store(torch.from_numpy(keys).cuda(), np.arange(300, dtype=np.uint32))
    snap = kt.save()
    torch.cuda.synchronize()
    assert kt.stamps.any()
    kt.load(snap)
    torch.cuda.synchronize()
    assert not kt.stamps.any()
    assert kt.entries() == 300
    kt.close()


_SEEDER = r'''
import sys
import numpy as np
import torch
sys.path.insert(0, sys.argv[1])
import __graft_entry__ as g
g.build()
from paper_2609_38706_gb300 import workloads as W
from paper_2609_38706_gb300.service import KeyTable
wl = W.reduced("multi_adapter")
b = wl.batch
kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
d = kt.digests(wl.descriptors)
key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
N = int(key_off[-1])
kt.store(keys[:N], np.arange(N, dtype=np.uint32) + 7000)
kt.check("seeder")
snap = torch.empty(kt.table.numel() + 64, dtype=torch.uint8).pin_memory()
kt.save(snap)
torch.cuda.synchronize()
np.save(sys.argv[2], snap.numpy())
'''


def test_seeder_and_retriever_in_separate_processes(tmp_path):
    """The paper's two-phase setup: a seeder process derives a batch's keys,
    stores them and saves the table; a retriever process loads the table and
    derives the keys again on its own.  Every request then hits in full with
    the seeder's slots, as the oracle's store-then-lookup says, and the same
    tokens under another salt hit nothing."""
    import os
    import subprocess
    import sys
    from paper_2609_38706_gb300.service import KeyTable, u32
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    path = str(tmp_path / "table.npy")
    subprocess.run([sys.executable, "-c", _SEEDER, root, path], check=True, timeout=600)
    wl = W.reduced("multi_adapter")
    b = wl.batch
    kt = KeyTable(wl.chunk_tokens, wl.capacity_log2)
    kt.load(torch.from_numpy(np.load(path)).pin_memory())
    d = kt.digests(wl.descriptors)
    key_off, keys = kt.derive(b.tokens, b.tok_off, b.desc_idx, d)
    hit, slots = kt.lookup(keys, key_off)
    kt.check("retriever")
    ko = key_off.cpu().numpy()
    N = int(ko[-1])
    dd = O.descriptor_digests(wl.descriptors)
    rko, rkeys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, dd)
    t = O.DictTable(wl.capacity)
    t.store(rkeys, np.arange(N, dtype=np.uint32) + 7000)
    rhit, rslots = O.lookup(t, rkeys, rko)
    assert np.array_equal(ko, rko)
    assert np.array_equal(hit.cpu().numpy(), rhit) and np.array_equal(rhit, np.diff(rko))
    assert np.array_equal(u32(slots)[:N], rslots)
    other = [dict(x, salt="another-domain") for x in wl.descriptors]
    ko2, keys2 = kt.derive(b.tokens, b.tok_off, b.desc_idx, kt.digests(other))
    hit2, _ = kt.lookup(keys2, ko2)
    kt.check("retriever, other salt")
    assert not hit2.cpu().numpy().any()
    kt.close()


def test_seeded_table_is_a_linear_probing_layout():
    """The device table is plain linear probing from the home entry (the first 8 key bytes, little-endian,
    modulo the capacity): every stored key lies at or after its home with no empty entry in between, and the
    mean successful probe length of the seeded multi-adapter table (2^20 entries at load 0.5) is Knuth's
    (1 + 1/(1 - a)) / 2 = 1.5 within 3% (a sanity check of the layout; results never depend on it)."""
    wl = W.FULL_CONFIGS["multi_adapter"]()
    kt, _ = _seeded(wl)
    e = kt.table.view(-1, 32).cpu().numpy()
    kt.close()
    cap = e.shape[0]
    mask = cap - 1
    occ = e[:, :16].any(axis=1)
    n = int(occ.sum())
    assert n == wl.target_entries
    home = e[:, :8].copy().view("<u8")[:, 0] & np.uint64(mask)
    dist = (np.arange(cap, dtype=np.uint64) - home) & np.uint64(mask)
    # length of the run of occupied entries ending at each entry, on a rotation that starts after an empty one
    shift = int(np.flatnonzero(~occ)[0]) + 1
    r = np.roll(occ, -shift)
    idx = np.arange(cap)
    last_empty = np.maximum.accumulate(np.where(~r, idx, -1))
    run = np.roll(idx - last_empty, shift)
    assert np.all(dist[occ] < run[occ].astype(np.uint64)), "a key is not reachable from its home"
    alpha = n / cap
    mean = float((dist[occ] + 1).mean())
    knuth = 0.5 * (1 + 1 / (1 - alpha))
    assert abs(mean - knuth) / knuth < 0.03, (mean, knuth)
