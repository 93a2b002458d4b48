"""Pins for the oracle's SHA-256 and chunk serialisation.

SHA-256 is checked against two references independent of the oracle: the
FIPS 180-2 Appendix B example digests (tests/golden) and Python's hashlib
(OpenSSL).  The little-endian int32 serialisation of a chunk is pinned by
re-expressing the published example messages as int32 tokens.
"""
import hashlib

import numpy as np
import pytest

import oracle as O


def test_published_examples(golden_sha256):
    assert len(golden_sha256) == 3
    for msg, digest in golden_sha256:
        assert O.sha256(msg) == digest


@pytest.mark.parametrize("length", range(0, 301))
def test_against_hashlib_every_length(length):
    # covers every padding boundary (55/56/63/64/119/120/127/128 bytes ...)
    rng = np.random.default_rng(length)
    msg = rng.integers(0, 256, length, dtype=np.uint8).tobytes()
    assert O.sha256(msg) == hashlib.sha256(msg).digest()


@pytest.mark.parametrize("length", [64, 96, 1024, 4 * 14, 4 * 255, 4 * 257, 1 << 20])
def test_against_hashlib_path_shapes(length):
    rng = np.random.default_rng(1000 + length)
    msg = rng.integers(0, 256, length, dtype=np.uint8).tobytes()
    assert O.sha256(msg) == hashlib.sha256(msg).digest()


def _as_le_tokens(msg: bytes) -> np.ndarray:
    assert len(msg) % 4 == 0
    return np.frombuffer(msg, dtype="<i4").astype(np.int32)


def test_chunk_serialisation_published_two_block(golden_sha256):
    # 56-byte FIPS example = 14 int32 tokens read little-endian
    msg, digest = golden_sha256[1]
    toks = _as_le_tokens(msg)
    assert toks.size == 14
    assert O.chunk_digest(toks) == digest
    # reading the same bytes big-endian gives different tokens -> different digest
    be = np.frombuffer(msg, dtype=">i4").astype(np.int32)
    assert O.chunk_digest(be) != digest


def test_chunk_serialisation_published_million_a(golden_sha256):
    msg, digest = golden_sha256[2]
    toks = _as_le_tokens(msg)
    assert toks.size == 250000 and np.all(toks == 0x61616161)
    assert O.chunk_digest(toks) == digest


def test_negative_and_extreme_tokens():
    toks = np.array([-1, -2**31, 2**31 - 1, 0, 1, 152063], dtype=np.int32)
    assert O.chunk_digest(toks) == hashlib.sha256(toks.astype("<i4").tobytes()).digest()


def test_constants_are_fips_values_by_digest():
    # The oracle derives K and H0 from their definitions; any wrong constant
    # changes the digest of the empty message.
    assert O.sha256(b"") == hashlib.sha256(b"").digest()
    k, h = O.constants()
    assert len(set(k.tolist())) == 64 and len(set(h.tolist())) == 8
