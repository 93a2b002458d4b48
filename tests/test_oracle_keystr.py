"""Pins of the oracle's connector key strings (Sec. 5.3, connector
integration: the 128-bit digest as twenty-two base64 characters, a
fixed-length hash over the model identity and worker provenance, a key whose
length does not depend on the model path).

The base64 encoder is pinned to the published test vectors of RFC 4648,
Sec. 10, and cross-checked against an independent implementation (the
standard library's); the 22-character form by its decoding and by the bit
layout the RFC fixes; the model tag and the row layout by their stated
structure."""
import base64

import numpy as np
import pytest

import oracle as O
from conftest import load_golden_base64

DESC = {"model_id": "org/model-7b", "weight_precision": "bf16", "weight_version": "rev-3",
        "adapter_id": "", "kv_format": "fp8_e4m3", "salt": ""}


@pytest.mark.parametrize("data,expected", load_golden_base64())
def test_base64_rfc4648_vectors(data, expected):
    assert O.base64_encode(data) == expected


def test_base64_matches_an_independent_encoder():
    rng = np.random.default_rng(1)
    for n in list(range(0, 40)) + [255, 256, 1000]:
        data = rng.integers(0, 256, n, dtype=np.uint8).tobytes()
        assert O.base64_encode(data) == base64.b64encode(data).decode("ascii")


def test_alphabet_indices():
    # RFC 4648 Table 1: value v -> A..Z (0-25), a..z (26-51), 0..9 (52-61), + (62), / (63)
    assert O.B64_ALPHABET[0] == "A" and O.B64_ALPHABET[25] == "Z" and O.B64_ALPHABET[26] == "a"
    assert O.B64_ALPHABET[51] == "z" and O.B64_ALPHABET[52] == "0" and O.B64_ALPHABET[61] == "9"
    assert O.B64_ALPHABET[62:] == "+/" and len(set(O.B64_ALPHABET)) == 64


def test_key_string_is_22_characters_that_decode_to_the_prefix():
    rng = np.random.default_rng(2)
    for _ in range(200):
        p = rng.integers(0, 256, 16, dtype=np.uint8).tobytes()
        s = O.key_string(p)
        assert len(s) == 22 and set(s) <= set(O.B64_ALPHABET)
        assert base64.b64decode(s + "==") == p
        assert O.B64_ALPHABET.index(s[-1]) & 15 == 0  # 2 data bits, 4 zero bits


def test_key_string_bit_layout():
    # single set bits: bit 0 (MSB of byte 0) is the top bit of the first
    # character; bit 127 (LSB of byte 15) is bit 4 of the last
    for bit in range(128):
        p = (1 << (127 - bit)).to_bytes(16, "big")
        s = O.key_string(p)
        q, r = divmod(bit, 6)
        expect = ["A"] * 22
        expect[q] = O.B64_ALPHABET[1 << (5 - r)]
        assert s == "".join(expect), bit
    assert O.key_string(bytes(16)) == "A" * 22
    assert O.key_string(b"\xff" * 16) == "/" * 21 + "w"


def test_key_string_is_injective_on_a_sample():
    rng = np.random.default_rng(3)
    ps = {rng.integers(0, 256, 16, dtype=np.uint8).tobytes() for _ in range(5000)}
    assert len({O.key_string(p) for p in ps}) == len(ps)


def test_key_string_rejects_other_lengths():
    for n in (0, 15, 17, 32):
        with pytest.raises(O.OracleError):
            O.key_string(bytes(n))


def test_model_tag_binds_worker_fields_only():
    base = O.model_tag(DESC)
    assert len(base) == 22 and base == O.key_string(O.worker_digest(DESC)[:16])
    for f, v in (("model_id", "org/model-8b"), ("weight_precision", "fp8"), ("weight_version", "rev-4"),
                 ("kv_format", "bf16")):
        assert O.model_tag({**DESC, f: v}) != base, f
    for f, v in (("adapter_id", "ad-1"), ("salt", "tenant-a")):
        assert O.model_tag({**DESC, f: v}) == base, f
    assert O.model_tag({**DESC, "weight_precision": "bfloat16"}) == base  # canonical spelling


def test_connector_key_length_does_not_depend_on_the_model_path():
    """Sec. 5.3: a 128-bit hex digest appended to an unbounded model path
    overruns a 150-byte field; the 22-character digest and the fixed-length
    model hash keep every key the same length."""
    rng = np.random.default_rng(4)
    keys = rng.integers(0, 256, (8, 32), dtype=np.uint8)
    lengths = set()
    for path_len in (1, 20, 150, 4000):
        desc = {**DESC, "model_id": "m" * path_len}
        prefix = ("fmt@" + O.model_tag(desc) + "@1@0@").encode()
        rows = O.key_strings(keys, prefix, 150)
        for row in rows:
            s = row.tobytes().rstrip(b"\0")
            lengths.add(len(s))
        hex_form = "fmt@" + desc["model_id"] + "@1@0@" + O.prefix128(keys)[0].tobytes().hex()
        assert (len(hex_form) > 150) == (path_len > 150 - 4 - 5 - 32)
    assert lengths == {4 + 22 + 5 + 22}


def test_key_strings_rows():
    rng = np.random.default_rng(5)
    keys = rng.integers(0, 256, (37, 32), dtype=np.uint8)
    rows = O.key_strings(keys, b"ab@", 64)
    assert rows.shape == (37, 64)
    for i in range(37):
        assert rows[i, :3].tobytes() == b"ab@"
        assert rows[i, 3:25].tobytes().decode() == O.key_string(keys[i, :16].tobytes())
        assert not rows[i, 25:].any()
    assert O.key_strings(keys[:0], b"", 22).shape == (0, 22)
    with pytest.raises(O.OracleError):
        O.key_strings(keys, b"x", 22)
