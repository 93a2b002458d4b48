"""Pins for descriptor canonicalisation, enc and the descriptor digest d.

enc must be injective (Sec. 5.2, Eq. 3): proven here by exhibiting a decoder
that recovers the field tuple from the bytes, over random tuples including
field-boundary shifts.  Canonicalisation binds resolved values only
(Sec. 5.3): ``auto`` and empty resolved fields are refused.  Extension
(Prop. 1): appending a field changes d and leaves existing registries alone.
"""
import hashlib
import subprocess
import sys

import numpy as np
import pytest

import oracle as O

BASE = {"model_id": "synthetic/model-7b", "weight_precision": "bf16", "weight_version": "v1",
        "adapter_id": "adapter-00", "kv_format": "bf16", "salt": "tenant-a"}


def decode(b: bytes):
    n = int.from_bytes(b[:4], "little")
    pos, out = 4, []
    for _ in range(n):
        ln = int.from_bytes(b[pos:pos + 4], "little")
        pos += 4
        out.append(b[pos:pos + ln])
        pos += ln
    assert pos == len(b)
    return tuple(out)


def test_enc_layout_small_case():
    e = O.enc((b"ab", b"", b"c"))
    assert e == bytes([3, 0, 0, 0, 2, 0, 0, 0]) + b"ab" + bytes(4) + bytes([1, 0, 0, 0]) + b"c"


def test_enc_boundary_shift():
    assert O.enc((b"ab", b"c")) != O.enc((b"a", b"bc"))
    assert O.enc((b"", b"abc")) != O.enc((b"abc", b""))
    assert O.enc((b"a",)) != O.enc((b"a", b""))


def test_enc_injective_random():
    rng = np.random.default_rng(7)
    seen = {}
    for _ in range(3000):
        n = int(rng.integers(0, 8))
        t = tuple(rng.integers(0, 3, int(rng.integers(0, 5)), dtype=np.uint8).tobytes() for _ in range(n))
        e = O.enc(t)
        assert decode(e) == t
        if e in seen:
            assert seen[e] == t
        seen[e] = t


def test_canonical_synonyms():
    for raw, canon in [("BF16", "bf16"), ("bfloat16", "bf16"), ("float16", "fp16"), ("half", "fp16"),
                       ("Float32", "fp32"), ("float", "fp32"), ("float8_e4m3fn", "fp8_e4m3"),
                       ("float8_e5m2", "fp8_e5m2")]:
        d = dict(BASE, weight_precision=raw, kv_format=raw)
        f = O.canonicalize(d)
        assert f[1] == canon.encode() and f[4] == canon.encode()
        assert O.descriptor_digest(d) == O.descriptor_digest(dict(BASE, weight_precision=canon,
                                                                   kv_format=canon))


def test_distinct_formats_never_merge():
    ds = {O.descriptor_digest(dict(BASE, kv_format=k)) for k in ("fp8", "fp8_e4m3", "fp8_e5m2", "bf16", "fp16")}
    assert len(ds) == 5


@pytest.mark.parametrize("field", ["weight_precision", "kv_format"])
@pytest.mark.parametrize("value", ["auto", "AUTO", "Auto", "", None])
def test_unresolved_refused(field, value):
    with pytest.raises(O.OracleError) as e:
        O.canonicalize(dict(BASE, **{field: value}))
    assert e.value.code == O.PK_ERR_UNRESOLVED


def test_opaque_fields_verbatim():
    f = O.canonicalize(dict(BASE, model_id="Org/Model", adapter_id="Adapter-A", salt="SaLt"))
    assert f[0] == b"Org/Model" and f[3] == b"Adapter-A" and f[5] == b"SaLt"
    assert O.descriptor_digest(dict(BASE, adapter_id="a")) != O.descriptor_digest(dict(BASE, adapter_id="A"))


def test_absent_equals_empty():
    d1 = dict(BASE, adapter_id="", salt="")
    d2 = {k: v for k, v in BASE.items() if k not in ("adapter_id", "salt")}
    assert O.descriptor_digest(d1) == O.descriptor_digest(d2)


def test_field_too_long():
    O.canonicalize(dict(BASE, salt="x" * O.MAX_FIELD_BYTES))
    with pytest.raises(O.OracleError) as e:
        O.canonicalize(dict(BASE, salt="x" * (O.MAX_FIELD_BYTES + 1)))
    assert e.value.code == O.PK_ERR_FIELD_TOO_LONG
    with pytest.raises(O.OracleError):
        O.canonicalize(dict(BASE, extra=[b"y" * (O.MAX_FIELD_BYTES + 1)]))


def test_every_field_changes_digest():
    d0 = O.descriptor_digest(BASE)
    for name in O.REGISTRY_V1:
        alt = "fp16" if name in ("weight_precision", "kv_format") else BASE[name] + "'"
        assert O.descriptor_digest(dict(BASE, **{name: alt})) != d0, name


def test_extension_prop1():
    d6 = O.descriptor_digest(BASE)
    d7 = O.descriptor_digest(dict(BASE, extra=[b"rope-base=1e6"]))
    d7b = O.descriptor_digest(dict(BASE, extra=[b"rope-base=5e5"]))
    d7e = O.descriptor_digest(dict(BASE, extra=[b""]))
    assert len({d6, d7, d7b, d7e}) == 4
    # the 6-field registry's encoding is untouched by the existence of extensions
    assert O.enc(O.canonicalize(BASE))[:4] == (6).to_bytes(4, "little")
    assert O.enc(O.canonicalize(dict(BASE, extra=[b"x"])))[:4] == (7).to_bytes(4, "little")


def test_digest_is_sha256_of_enc():
    e = O.enc(O.canonicalize(BASE))
    assert O.descriptor_digest(BASE) == hashlib.sha256(e).digest()


def test_cross_worker_stability():
    code = ("import sys; sys.path.insert(0, %r); import oracle as O; "
            "print(O.descriptor_digest(%r).hex())") % (O.__file__.rsplit("/oracle/", 1)[0], BASE)
    outs = {subprocess.check_output([sys.executable, "-c", code], text=True).strip() for _ in range(2)}
    assert outs == {O.descriptor_digest(BASE).hex()}
