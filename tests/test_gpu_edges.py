"""GPU edge cases and error paths, each checked against the oracle or against
the documented status codes.  Every failure here is produced on the host or
by the kernels' own bounds checks: nothing faults, traps or waits unboundedly."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_38706_gb300 import pk
from paper_2609_38706_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DESC = {"model_id": "synthetic/model-7b", "weight_precision": "bf16", "weight_version": "v1",
        "adapter_id": "adapter-00", "kv_format": "bf16", "salt": ""}


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")


def KT(C=16, log2=8, max_probe=0):
    from paper_2609_38706_gb300.service import KeyTable
    return KeyTable(C, log2, max_probe)


def derive_both(kt, rows, desc_idx, descs, C):
    toks = np.concatenate([np.asarray(r, np.int32) for r in rows]) if rows else np.zeros(0, np.int32)
    off = np.zeros(len(rows) + 1, np.int64)
    np.cumsum([len(r) for r in rows], out=off[1:])
    d = kt.digests(descs)
    ko, keys = kt.derive(toks, off, np.asarray(desc_idx, np.uint32), d)
    kt.check("derive")
    rko, rkeys = O.derive_keys(toks, off, C, np.asarray(desc_idx, np.uint32), O.descriptor_digests(descs))
    N = int(ko[-1].item()) if ko.numel() else 0
    return ko.cpu().numpy(), keys.cpu().numpy()[:N], rko, rkeys


@pytest.mark.parametrize("C", [1, 2, 3, 4, 5, 13, 14, 15, 16, 17, 31, 64, 100, 255, 256, 257, 1000])
def test_chunk_sizes_and_unaligned_starts(C):
    rng = np.random.default_rng(C)
    rows = [rng.integers(-2**31, 2**31, int(rng.integers(0, 4 * C + 3)), dtype=np.int64).astype(np.int32)
            for _ in range(37)]
    kt = KT(C)
    ko, keys, rko, rkeys = derive_both(kt, rows, rng.integers(0, 2, 37), [DESC, dict(DESC, salt="t")], C)
    assert np.array_equal(ko, rko) and np.array_equal(keys, rkeys)
    kt.close()


@pytest.mark.parametrize("C", [21, 30])
def test_multiply_add_round_form_with_ragged_unaligned_requests(C):
    """A batch of more than 3 x 4 x 32 x 152 = 58,368 chunks, so that the
    chunk digests run in the multiply-add round form, with requests of random
    token counts (unaligned starts: 16-byte token loads and plain loads), and
    chunk sizes whose final block holds tokens and the padding (C = 21, 5
    tokens and the length in one block) or spills the length into a second
    padding block (C = 30, 14 tokens)."""
    rng = np.random.default_rng(1000 + C)
    R = 6000
    rows = [rng.integers(-2**31, 2**31, int(rng.integers(0, 40 * C)), dtype=np.int64).astype(np.int32)
            for _ in range(R)]
    assert sum(len(r) // C for r in rows) > 58_368
    kt = KT(C)
    ko, keys, rko, rkeys = derive_both(kt, rows, rng.integers(0, 2, R), [DESC, dict(DESC, adapter_id="a1")], C)
    assert np.array_equal(ko, rko) and np.array_equal(keys, rkeys)
    kt.close()


def test_published_vector_chunks():
    # FIPS 180-2 B.3 message (10^6 'a') as one 250000-token chunk, and B.2 as one 14-token chunk.
    a = np.full(250000, 0x61616161, np.int32)
    b = np.frombuffer(b"abcdbcdecdefdefgefghfghighijhijkijkljklmklmnlmnomnopnopq", "<i4").astype(np.int32)
    for C, row in ((250000, a), (14, b)):
        kt = KT(C)
        ko, keys, rko, rkeys = derive_both(kt, [row, row], [0, 0], [DESC], C)
        assert np.array_equal(keys, rkeys) and keys.shape[0] == 2
        kt.close()


def test_empty_batch_and_empty_requests():
    kt = KT(16)
    ko, keys, rko, rkeys = derive_both(kt, [], [], [DESC], 16)
    assert ko.tolist() == [0] and keys.shape[0] == 0
    ko, keys, rko, rkeys = derive_both(kt, [[], [1] * 15, []], [0, 0, 0], [DESC], 16)
    assert ko.tolist() == [0, 0, 0, 0] and keys.shape[0] == 0
    # lookup / store of zero keys
    key_off = torch.zeros(4, dtype=torch.int64, device="cuda")
    hit, slots = kt.lookup(torch.zeros((0, 32), dtype=torch.uint8, device="cuda"), key_off)
    assert hit.cpu().tolist() == [0, 0, 0]
    res, so = kt.store(torch.zeros((0, 32), dtype=torch.uint8, device="cuda"), np.zeros(0, np.uint32))
    kt.check()
    kt.close()


def test_bad_offsets_report_and_produce_no_keys():
    kt = KT(16)
    d = kt.digests([DESC])
    toks = np.arange(64, dtype=np.int32)
    for off, idx in (([0, 32, 16, 64], [0, 0, 0]),      # decreasing
                     ([0, 32, 80], [0, 0]),             # beyond n_tokens
                     ([-4, 32, 64], [0, 0]),            # negative
                     ([0, 32, 64], [0, 1])):            # descriptor index out of range
        ko, keys = kt.derive(toks, np.array(off, np.int64), np.array(idx, np.uint32), d)
        assert kt.take_status() == pk.PK_ERR_ARG
        assert ko.cpu().numpy().tolist() == [0] * len(off)
    kt.close()


def test_host_argument_errors():
    kt = KT(16)
    d = kt.digests([DESC])
    toks = torch.arange(64, dtype=torch.int32, device="cuda")
    off = torch.tensor([0, 64], dtype=torch.int64, device="cuda")
    idx = torch.zeros(1, dtype=torch.int32, device="cuda")
    ko = torch.empty(2, dtype=torch.int64, device="cuda")
    small = torch.empty((3, 32), dtype=torch.uint8, device="cuda")      # needs 4 keys
    with pytest.raises(pk.PKError) as e:
        pk.pk_derive_keys(kt.ctx, toks, off, idx, d, ko, small, kt.status)
    assert e.value.code == pk.PK_ERR_ARG
    buf = torch.empty(4 * 32 + 8, dtype=torch.uint8, device="cuda")
    misaligned = buf[8:].view(4, 32)                                      # 8-byte offset
    with pytest.raises(pk.PKError):
        pk.pk_derive_keys(kt.ctx, toks, off, idx, d, ko, misaligned, kt.status)
    with pytest.raises(pk.PKError):
        pk.pk_store(kt.ctx, misaligned, torch.zeros(4, dtype=torch.int32, device="cuda"),
                    torch.empty(4, dtype=torch.int32, device="cuda"), torch.empty(4, dtype=torch.int32, device="cuda"),
                    kt.status, key_off=off)                              # key_off without hit_chunks
    with pytest.raises(pk.PKError) as e:
        KT(16, log2=0)
    assert e.value.code == pk.PK_ERR_CAPACITY
    kt.close()


def _keys16(vals):
    k = np.zeros((len(vals), 16), np.uint8)
    for i, v in enumerate(vals):
        k[i] = np.frombuffer(int(v).to_bytes(16, "little"), np.uint8)
    return k


def test_duplicates_lowest_index_wins_under_contention():
    rng = np.random.default_rng(1)
    pool = _keys16(rng.integers(1, 2**62, 50, dtype=np.int64))
    keys = pool[rng.integers(0, 50, 20000)]
    slots = rng.integers(0, 2**32 - 1, 20000, dtype=np.uint64).astype(np.uint32)
    kt = KT(16, log2=10)
    res, so = kt.store(keys, slots)
    kt.check()
    t = O.DictTable(1024)
    rres, rso = t.store(keys, slots)
    assert np.array_equal(res.cpu().numpy(), rres)
    assert np.array_equal(so.cpu().numpy().view(np.uint32), rso)
    assert kt.entries() == len(t) == 50
    # a second call sees them as pre-existing
    res2, so2 = kt.store(keys[:100], slots[:100] ^ 1)
    rres2, rso2 = t.store(keys[:100], slots[:100] ^ 1)
    assert np.array_equal(res2.cpu().numpy(), rres2) and np.array_equal(so2.cpu().numpy().view(np.uint32), rso2)
    kt.close()


def test_same_home_collisions():
    # 40 keys sharing their first 8 bytes (same home entry) -> one long probe run
    base = _keys16([1 << 70])
    keys = np.repeat(base, 40, axis=0)
    keys[:, 8] = np.arange(40)
    keys[:, 9] = 7
    slots = np.arange(40, dtype=np.uint32)
    kt = KT(16, log2=8)
    res, so = kt.store(keys, slots)
    kt.check()
    assert (res.cpu().numpy() == pk.PK_STORE_INSERTED).all()
    key_off = torch.tensor([0, 40], dtype=torch.int64, device="cuda")
    k32 = torch.zeros((40, 32), dtype=torch.uint8, device="cuda")
    k32[:, :16] = torch.from_numpy(keys).cuda()
    hit, got = kt.lookup(k32, key_off)
    kt.check()
    assert hit.cpu().tolist() == [40] and got.cpu().numpy().tolist() == slots.tolist()
    kt.close()


def test_table_full_and_probe_limit_report_without_hanging():
    kt = KT(16, log2=3)                         # 8 entries: at most 7 stored
    res, _ = kt.store(_keys16(range(1, 8)), np.arange(7, dtype=np.uint32))
    kt.check()
    assert kt.entries() == 7
    res, so = kt.store(_keys16([100, 101, 3]), np.array([9, 9, 9], np.uint32))
    assert kt.take_status() == pk.PK_ERR_TABLE_FULL
    assert res.cpu().tolist() == [pk.PK_ERR_TABLE_FULL, pk.PK_ERR_TABLE_FULL, pk.PK_STORE_PRESENT]
    assert kt.entries() == 7
    kt.close()

    kt = KT(16, log2=8, max_probe=1)
    base = _keys16([5, 5 + (1 << 64)])          # same home, different keys
    res, _ = kt.store(base, np.array([1, 2], np.uint32))
    assert kt.take_status() == pk.PK_ERR_PROBE_LIMIT
    assert sorted(res.cpu().tolist()) == [pk.PK_ERR_PROBE_LIMIT, pk.PK_STORE_INSERTED]
    k32 = torch.zeros((2, 32), dtype=torch.uint8, device="cuda")
    k32[:, :16] = torch.from_numpy(base).cuda()
    hit, slots = kt.lookup(k32, torch.tensor([0, 2], dtype=torch.int64, device="cuda"))
    assert kt.take_status() == pk.PK_ERR_PROBE_LIMIT
    kt.close()


def test_reserved_key_and_reserved_slot():
    kt = KT(16, log2=6)
    keys = _keys16([0, 9, 10])
    res, so = kt.store(keys, np.array([1, pk.PK_NO_SLOT, 3], np.uint32))
    assert kt.take_status() in (pk.PK_ERR_RESERVED_KEY, pk.PK_ERR_ARG)
    assert res.cpu().tolist() == [pk.PK_ERR_RESERVED_KEY, pk.PK_ERR_ARG, pk.PK_STORE_INSERTED]
    k32 = torch.zeros((3, 32), dtype=torch.uint8, device="cuda")
    k32[:, :16] = torch.from_numpy(keys).cuda()
    hit, slots = kt.lookup(k32, torch.tensor([0, 3], dtype=torch.int64, device="cuda"))
    kt.check()
    assert hit.cpu().tolist() == [0]
    assert slots.cpu().numpy().view(np.uint32).tolist() == [pk.PK_NO_SLOT, pk.PK_NO_SLOT, 3]
    kt.close()


def test_descriptor_digest_device_equals_host_and_oracle():
    rng = np.random.default_rng(9)
    descs = []
    for j in range(64):
        d = dict(DESC, weight_version=bytes(rng.integers(0, 256, j * 13, dtype=np.uint8)), salt="s%d" % j)
        if j % 3 == 0:
            d["extra"] = [b"x" * j]
        descs.append(d)
    kt = KT(16)
    dg = kt.digests(descs).cpu().numpy()
    kt.check()
    assert np.array_equal(dg, O.descriptor_digests(descs))
    assert all(pk.pk_descriptor_digest(d) == dg[j].tobytes() for j, d in enumerate(descs))
    kt.close()


@pytest.mark.parametrize("R,C", [(9000, 16), (5000, 7)])
def test_many_requests_span_scan_tiles_and_parts(R, C):
    """More requests than one scan tile (4096), many chunks; ragged lengths
    and empty requests."""
    rng = np.random.default_rng(R + C)
    lens = rng.integers(0, 40 * C, R)
    lens[::13] = 0
    rows = [rng.integers(0, 152064, int(n)).astype(np.int32) for n in lens]
    descs = [DESC, dict(DESC, salt="a"), dict(DESC, adapter_id="adapter-07")]
    kt = KT(C, log2=10)
    ko, keys, rko, rkeys = derive_both(kt, rows, rng.integers(0, 3, R), descs, C)
    assert np.array_equal(ko, rko) and np.array_equal(keys, rkeys)
    kt.close()


@pytest.mark.parametrize("layout", ["uniform", "skewed", "empty_runs"])
def test_chunk_to_request_mapping_paths(layout):
    """The chunk-digest warps map their 32 chunks to requests from a guess
    (requests of about equal size), checked against 32 loaded offsets, and fall
    back to a search when the guess misses or the window ends inside a run of
    empty requests.  Uniform requests take the guess; a skewed batch (a few
    huge requests among small ones) misses it; runs of 40-200 empty requests
    between short ones end the window early.  Keys compared with the oracle."""
    rng = np.random.default_rng({"uniform": 1, "skewed": 2, "empty_runs": 3}[layout])
    C = 16
    if layout == "uniform":
        lens = np.full(3000, 8 * C, np.int64)
    elif layout == "skewed":
        lens = rng.integers(0, 3 * C, 3000)
        lens[rng.integers(0, 3000, 12)] = rng.integers(200 * C, 400 * C, 12)
    else:
        lens = np.zeros(6000, np.int64)
        i = 0
        while i < lens.size:
            lens[i] = rng.integers(1, 6 * C)
            i += 1 + int(rng.integers(40, 200)) if rng.random() < 0.3 else 1
    rows = [rng.integers(0, 152064, int(n)).astype(np.int32) for n in lens]
    kt = KT(C, log2=10)
    ko, keys, rko, rkeys = derive_both(kt, rows, rng.integers(0, 2, lens.size), [DESC, dict(DESC, salt="m")], C)
    assert np.array_equal(ko, rko) and np.array_equal(keys, rkeys)
    kt.close()
