"""Pins of the oracle's content identity (Sec. 5.3 adapter identity; Sec. 5.1:
injective and stable): the fixed-shape SHA-256 tree checked against hashlib
built by hand for one, two and three levels, its shape, and the properties the
identity needs (the byte length and every tensor attribute bound)."""
import hashlib

import numpy as np
import pytest

import oracle as O


def H(b: bytes) -> bytes:
    return hashlib.sha256(b).digest()


def blocks(b: bytes):
    n = max(1, -(-len(b) // 1024))
    b = b + bytes(n * 1024 - len(b))
    return [b[i * 1024:(i + 1) * 1024] for i in range(n)]


@pytest.mark.parametrize("n", [0, 1, 55, 1023, 1024])
def test_one_block_is_sha256_of_the_zero_padded_block(n):
    data = bytes(np.random.default_rng(n).integers(0, 256, n, dtype=np.uint8))
    assert O.content_digest(data) == H(data + bytes(1024 - n))


def test_two_and_three_levels_by_hand():
    rng = np.random.default_rng(4)
    data = bytes(rng.integers(0, 256, 3000, dtype=np.uint8))          # 3 leaves, one node
    leaves = b"".join(H(x) for x in blocks(data))
    assert O.content_digest(data) == H(leaves + bytes(1024 - len(leaves)))
    data = bytes(rng.integers(0, 256, 33 * 1024 + 1, dtype=np.uint8))  # 34 leaves -> 2 nodes -> top
    l1 = b"".join(H(x) for x in blocks(data))
    l2 = b"".join(H(x) for x in blocks(l1))
    assert len(l1) == 34 * 32 and len(l2) == 64
    assert O.content_digest(data) == H(l2 + bytes(1024 - 64))


def test_every_byte_matters_and_the_length_is_bound_by_the_identity():
    rng = np.random.default_rng(5)
    data = bytearray(rng.integers(0, 256, 70_000, dtype=np.uint8))
    top = O.content_digest(bytes(data))
    for pos in (0, 1023, 1024, 50_000, 69_999):
        d2 = bytearray(data)
        d2[pos] ^= 0x01
        assert O.content_digest(bytes(d2)) != top, pos
    # zero padding is invisible to the tree, not to the identity (the length is bound)
    assert O.content_digest(bytes(data) + b"\0") == top
    assert O.tensor_identity("w", "bf16", [35000], 70_000, top) != O.tensor_identity("w", "bf16", [35000], 70_001, top)


def test_identity_binds_name_dtype_shape_and_the_adapter_binds_order_and_config():
    top = O.content_digest(b"x" * 100)
    base = O.tensor_identity("layers.0.q", "bf16", [10, 5], 100, top)
    assert base != O.tensor_identity("layers.0.k", "bf16", [10, 5], 100, top)
    assert base != O.tensor_identity("layers.0.q", "fp16", [10, 5], 100, top)
    assert base != O.tensor_identity("layers.0.q", "bf16", [5, 10], 100, top)
    assert base != O.tensor_identity("layers.0.q", "bf16", [50], 100, top)
    other = O.tensor_identity("layers.1.q", "bf16", [10, 5], 100, top)
    a = O.adapter_identity([base, other], ["r=8", "alpha=16"])
    assert a != O.adapter_identity([other, base], ["r=8", "alpha=16"])
    assert a != O.adapter_identity([base, other], ["r=16", "alpha=16"])
    assert a != O.adapter_identity([base, other], ["r=8alpha=16"])
    assert a == O.adapter_identity([base, other], ["r=8", "alpha=16"])   # stable
