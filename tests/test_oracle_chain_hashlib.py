"""Pin of the oracle's key chain (C, FIPS 180-4 written out) against a second,
independent implementation built on the standard library's SHA-256
(hashlib / OpenSSL), over ragged batches of several configurations."""
import numpy as np
import pytest

import oracle as O
from paper_2609_38706_gb300 import workloads as W


@pytest.mark.parametrize("name", ["tiny", "multi_adapter", "small_block", "long_context", "provenance_sweep_D4"])
def test_c_chain_equals_hashlib_chain(name):
    wl = W.reduced(name)
    b = wl.batch
    d = O.descriptor_digests(wl.descriptors)
    ko, keys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d)
    R = b.R
    pick = list(range(R)) if R <= 64 else list(np.random.default_rng(0).choice(R, 64, replace=False))
    want = np.concatenate([keys[ko[r]:ko[r + 1]] for r in pick]) if pick else keys[:0]
    assert np.array_equal(O.derive_keys_hashlib(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d, pick), want)


def test_chunk_size_one_and_partial_chunks():
    rng = np.random.default_rng(5)
    toks = rng.integers(-2**31, 2**31 - 1, 37, dtype=np.int64).astype(np.int32)
    d = bytes(range(32))
    for C in (1, 3, 16, 36, 37, 38):
        assert np.array_equal(O.request_keys_hashlib(toks, C, d), O.request_keys(toks, C, d))
