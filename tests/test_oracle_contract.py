"""Pins for the oracle's chained keys: the contract's invariants by brute force.

* Computational / permission invariants (Eqs. 1 and 2) and the differential
  omission test (Eq. 4): changing any one registered dimension, the salt
  included, changes every key of a request.
* Cross-worker stability (Sec. 5.1): identical tokens and descriptor give
  identical keys in another process and in another batch layout.
* Prefix structure of the chain: a changed token in chunk j changes keys
  j.. and leaves keys ..j-1 alone (catches dropped k_{i-1}, dropped c_i and
  off-by-one chunk indexing).
* Full chunks only (Sec. 4.4): floor(T / C) keys per request.
* Table 2 / Table 3 structures at key level.
"""
import hashlib
import subprocess
import sys

import numpy as np
import pytest

import oracle as O
from paper_2609_38706_gb300 import workloads as W

BASE = {"model_id": "synthetic/model-7b", "weight_precision": "bf16", "weight_version": "v1",
        "adapter_id": "adapter-00", "kv_format": "bf16", "salt": ""}
C = 16


def keys_of(tokens, desc, C=C):
    return O.request_keys(np.asarray(tokens, np.int32), C, O.descriptor_digest(desc))


@pytest.fixture(scope="module")
def toks():
    return np.random.default_rng(11).integers(0, 152064, 5 * C + 7).astype(np.int32)


def test_full_chunks_only(toks):
    k = keys_of(toks, BASE)
    assert k.shape == (5, 32)
    assert keys_of(toks[: C - 1], BASE).shape == (0, 32)
    assert keys_of(toks[:C], BASE).shape == (1, 32)
    # the partial tail does not influence any key
    t2 = toks.copy()
    t2[5 * C:] += 1
    assert np.array_equal(keys_of(t2, BASE), k)


@pytest.mark.parametrize("field", O.REGISTRY_V1)
def test_any_field_changes_every_key(toks, field):
    alt = "fp16" if field in ("weight_precision", "kv_format") else BASE[field] + "x"
    k0 = keys_of(toks, BASE)
    k1 = keys_of(toks, dict(BASE, **{field: alt}))
    assert np.all(np.any(k0 != k1, axis=1)), field


def test_extension_changes_every_key(toks):
    k0 = keys_of(toks, BASE)
    k1 = keys_of(toks, dict(BASE, extra=[b"rope-base"]))
    assert np.all(np.any(k0 != k1, axis=1))


@pytest.mark.parametrize("j", range(5))
def test_changed_chunk_changes_suffix_only(toks, j):
    k0 = keys_of(toks, BASE)
    for pos in (j * C, j * C + C // 2, j * C + C - 1):
        t = toks.copy()
        t[pos] ^= 1
        k1 = keys_of(t, BASE)
        assert np.array_equal(k1[:j], k0[:j])
        assert np.all(np.any(k1[j:] != k0[j:], axis=1))


def test_identical_inputs_identical_keys_across_layouts():
    wl = W.reduced("multi_adapter")
    d = O.descriptor_digests(wl.descriptors)
    b = wl.batch
    ko, keys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d)
    perm = np.random.default_rng(3).permutation(b.R)
    pb = b.select(perm)
    ko2, keys2 = O.derive_keys(pb.tokens, pb.tok_off, wl.chunk_tokens, pb.desc_idx, d)
    for new_r, old_r in enumerate(perm):
        assert np.array_equal(keys2[ko2[new_r]:ko2[new_r + 1]], keys[ko[old_r]:ko[old_r + 1]])
    # batch form == per-request form
    for r in range(b.R):
        kr = O.request_keys(b.tokens[b.tok_off[r]:b.tok_off[r + 1]], wl.chunk_tokens, d[b.desc_idx[r]].tobytes())
        assert np.array_equal(kr, keys[ko[r]:ko[r + 1]])


def test_identical_keys_across_processes(toks):
    root = O.__file__.rsplit("/oracle/", 1)[0]
    code = ("import sys, numpy as np; sys.path.insert(0, %r); import oracle as O; "
            "t = np.array(%r, np.int32); print(O.request_keys(t, %d, O.descriptor_digest(%r)).tobytes().hex())"
            % (root, toks.tolist(), C, BASE))
    outs = {subprocess.check_output([sys.executable, "-c", code], text=True).strip() for _ in range(2)}
    assert outs == {keys_of(toks, BASE).tobytes().hex()}


def test_threads_do_not_change_keys():
    wl = W.reduced("small_block")
    d = O.descriptor_digests(wl.descriptors)
    b = wl.batch
    n0 = O.max_threads()
    try:
        O.set_threads(1)
        _, k1 = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d)
        O.set_threads(max(n0, 4))
        _, k4 = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d)
    finally:
        O.set_threads(n0)
    assert np.array_equal(k1, k4)


def test_chain_against_hashlib_definition(toks):
    # An independent SHA-256 (OpenSSL) evaluating the stated definition.
    d = O.descriptor_digest(BASE)
    prev = bytes(32)
    expect = []
    for i in range(len(toks) // C):
        c = hashlib.sha256(toks[i * C:(i + 1) * C].astype("<i4").tobytes()).digest()
        prev = hashlib.sha256(prev + d + c).digest()
        expect.append(prev)
    assert keys_of(toks, BASE).tobytes() == b"".join(expect)


def test_key_count_closed_form():
    for name in ("multi_adapter", "small_block", "long_context", "provenance_sweep_D4"):
        wl = W.reduced(name)
        d = O.descriptor_digests(wl.descriptors)
        b = wl.batch
        ko, keys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d)
        lens = np.diff(b.tok_off)
        assert keys.shape[0] == int((lens // wl.chunk_tokens).sum()) == ko[-1]


# ---- Table 2 (paired matrix) and Table 3 (adapter x salt) at key level -------------------------
def _hit(seed_desc, probe_desc, toks):
    t = O.DictTable(64)
    ks = keys_of(toks, seed_desc)
    t.store(ks, np.arange(ks.shape[0]))
    kp = keys_of(toks, probe_desc)
    hit, _ = O.lookup(t, kp, np.array([0, kp.shape[0]]))
    return int(hit[0])


def test_table2_cases(toks):
    n = len(toks) // C
    miss_cases = [dict(weight_version="v2"), dict(weight_precision="fp8_e4m3"), dict(kv_format="fp16"),
                  dict(kv_format="fp8_e5m2"), dict(weight_version="v2", kv_format="fp16"),
                  dict(adapter_id="adapter-00@sha256:other-bytes"), dict(salt="tenant-b"),
                  dict(adapter_id="adapter-01"), dict(adapter_id="adapter-01", salt="tenant-b")]
    for ch in miss_cases:
        assert _hit(BASE, dict(BASE, **ch), toks) == 0, ch
    # same provenance, and the same adapter identity bytes reached through another path
    assert _hit(BASE, dict(BASE), toks) == n
    assert _hit(BASE, dict(BASE, adapter_id=str(BASE["adapter_id"])), toks) == n


def test_table3_adapter_salt_grid(toks):
    n = len(toks) // C
    seed = dict(BASE, adapter_id="A", salt="s1")
    grid = {(a, s): _hit(seed, dict(BASE, adapter_id=a, salt=s), toks)
            for a in ("A", "B") for s in ("s1", "s2")}
    assert grid == {("A", "s1"): n, ("A", "s2"): 0, ("B", "s1"): 0, ("B", "s2"): 0}
