"""Pins of the oracle's store-side omission test (Sec. 6.3; Eq. 4): the join
and page comparison against brute force over all key pairs and against its
special cases, and the experiment's shape in miniature: omitting a dimension
the two workers differ in, and that changes the cached state, flags every
shared page; the complete binding flags none; a salt changes keys, not state."""
import numpy as np
import pytest

import oracle as O
from paper_2609_38706_gb300 import workloads as W


def brute(ref_keys, ref_pages, keys, pages):
    v = np.zeros(keys.shape[0], np.int32)
    for j in range(keys.shape[0]):
        for i in range(ref_keys.shape[0]):          # first reference page with the same 16-byte prefix
            if bytes(ref_keys[i, :16]) == bytes(keys[j, :16]):
                v[j] = O.PAGE_EQUAL if bytes(ref_pages[i]) == bytes(pages[j]) else O.PAGE_DIFFERS
                break
    return v


@pytest.mark.parametrize("seed", range(6))
def test_join_and_compare_equal_brute_force(seed):
    rng = np.random.default_rng(seed)
    pool = rng.integers(0, 256, (12, 32), dtype=np.uint8)
    pool[:, 0] |= 1
    ref_keys = pool[rng.integers(0, 12, 20)]                 # repeated keys: the first one is the reference
    keys = pool[rng.integers(0, 12, 25)].copy()
    keys[:3, 20:] ^= 0xFF                                     # bytes past the 16-byte prefix do not matter
    ref_pages = rng.integers(0, 3, (20, 32), dtype=np.uint8)  # few values: equal pages happen
    pages = rng.integers(0, 3, (25, 32), dtype=np.uint8)
    v, counts = O.omission_check(ref_keys, ref_pages, keys, pages)
    assert np.array_equal(v, brute(ref_keys, ref_pages, keys, pages))
    assert counts.tolist() == np.bincount(v, minlength=3).tolist()


def test_special_cases():
    rng = np.random.default_rng(9)
    keys = rng.integers(1, 256, (40, 32), dtype=np.uint8)
    pages = rng.integers(0, 256, (40, 64), dtype=np.uint8)
    v, c = O.omission_check(keys, pages, keys, pages)             # a worker against itself
    assert (v == O.PAGE_EQUAL).all() and c.tolist() == [0, 40, 0]
    other = keys.copy()
    other[:, 0] ^= 0x80                                            # disjoint keys
    v, c = O.omission_check(keys, pages, other, pages)
    assert (v == O.PAGE_ABSENT).all()
    flipped = pages.copy()
    flipped[17, 63] ^= 1                                           # one byte of one page
    v, c = O.omission_check(keys, pages, keys, flipped)
    assert np.nonzero(v == O.PAGE_DIFFERS)[0].tolist() == [17] and c.tolist() == [0, 39, 1]


def test_pages_follow_prefix_and_computational_dimensions():
    case = W.omission_case("weight_version", None)
    b, C = case.batch, case.chunk_tokens
    pa = W.kv_pages(b, C, lambda r: case.worker_a, 64)
    assert np.array_equal(pa, W.kv_pages(b, C, lambda r: dict(case.worker_a, salt="other"), 64))   # salt: same state
    for f, v in (("weight_version", "x"), ("kv_format", "fp16"), ("adapter_id", "a9"), ("weight_precision", "fp16"),
                 ("model_id", "m2")):
        pb = W.kv_pages(b, C, lambda r: dict(case.worker_a, **{f: v}), 64)
        assert not np.any(np.all(pa == pb, axis=1)), f


@pytest.mark.parametrize("varied", ["model_id", "weight_precision", "weight_version", "adapter_id", "kv_format"])
def test_omitting_a_state_changing_dimension_flags_every_page(varied):
    for omit, expect in ((None, "none"), (varied, "all")):
        case = W.omission_case(varied, omit)
        b, C = case.batch, case.chunk_tokens
        _, ka = O.derive_keys(b.tokens, b.tok_off, C, b.desc_idx, O.descriptor_digests([case.bound_a]))
        _, kb = O.derive_keys(b.tokens, b.tok_off, C, b.desc_idx, O.descriptor_digests([case.bound_b]))
        v, counts = O.omission_check(ka, case.pages_a, kb, case.pages_b)
        n = ka.shape[0]
        assert counts.tolist() == ([n, 0, 0] if expect == "none" else [0, 0, n]), (varied, omit)


def test_salt_omission_is_not_a_state_collision():
    case = W.omission_case("salt", "salt")
    b, C = case.batch, case.chunk_tokens
    _, ka = O.derive_keys(b.tokens, b.tok_off, C, b.desc_idx, O.descriptor_digests([case.bound_a]))
    _, kb = O.derive_keys(b.tokens, b.tok_off, C, b.desc_idx, O.descriptor_digests([case.bound_b]))
    v, counts = O.omission_check(ka, case.pages_a, kb, case.pages_b)
    assert counts.tolist() == [0, ka.shape[0], 0]
