"""C-ABI checks that need no GPU: the library loads, exports every entry point
include/pk.h declares, and its host-side steps (descriptor canonicalisation,
enc and the descriptor digest d of Eq. 3) match the oracle exactly; host
argument errors are reported before any CUDA call."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle as O
from paper_2609_38706_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def pk():
    _build.build()
    from paper_2609_38706_gb300 import pk as pk_mod
    pk_mod.lib()
    return pk_mod


def declared_functions():
    src = open(os.path.join(ROOT, "include", "pk.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pk_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("pk_init", "pk_derive_keys", "pk_lookup", "pk_store", "pk_destroy", "pk_descriptor_digest"):
        assert required in names


def test_library_exports_every_declared_symbol(pk):
    L = ctypes.CDLL(_build.LIB)
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert not missing, missing


def test_status_vocabulary_matches_header(pk):
    src = open(os.path.join(ROOT, "include", "pk.h")).read()
    for name in ("PK_ERR_ARG", "PK_ERR_CAPACITY", "PK_ERR_UNRESOLVED", "PK_ERR_FIELD_TOO_LONG", "PK_ERR_TABLE_FULL",
                 "PK_ERR_PROBE_LIMIT", "PK_ERR_RESERVED_KEY", "PK_STORE_INSERTED", "PK_STORE_PRESENT"):
        m = re.search(r"#define %s \(?(-?\d+)\)?" % name, src)
        assert m and int(m.group(1)) == getattr(pk, name) == getattr(O, name.replace("PK_STORE_", "STORE_"), getattr(pk, name))


def _rand_desc(rng):
    pick = lambda opts: opts[int(rng.integers(0, len(opts)))]
    d = {"model_id": pick(["synthetic/model-7b", "Org/Model", "", "m" * 300]),
         "weight_precision": pick(["bf16", "BF16", "bfloat16", "fp8", "fp8_e4m3", "float8_e4m3fn", "Half", "int4-awq"]),
         "weight_version": bytes(rng.integers(0, 256, int(rng.integers(0, 50)), dtype=np.uint8)),
         "adapter_id": pick(["", "adapter-00", "Adapter-00", "sha256:" + "ab" * 32]),
         "kv_format": pick(["bf16", "fp16", "float16", "fp8_e5m2", "FP8_E4M3", "float32"]),
         "salt": pick(["", "tenant-a", "été"])}
    if rng.random() < 0.3:
        d["extra"] = [bytes(rng.integers(0, 256, int(rng.integers(0, 9)), dtype=np.uint8))
                      for _ in range(int(rng.integers(1, 4)))]
    return d


def test_descriptor_digest_matches_oracle(pk):
    rng = np.random.default_rng(5)
    for _ in range(500):
        d = _rand_desc(rng)
        assert pk.pk_descriptor_encode(d) == O.enc(O.canonicalize(d))
        assert pk.pk_descriptor_digest(d) == O.descriptor_digest(d)


def test_two_level_digests_match_oracle(pk):
    rng = np.random.default_rng(15)
    for _ in range(500):
        d = _rand_desc(rng)
        w = pk.pk_worker_digest(d)
        assert w == O.worker_digest(d)
        assert pk.pk_request_digest(w, d) == O.request_digest(w, d)
        other = bytes(rng.integers(0, 256, 32, dtype=np.uint8))  # any worker digest composes
        assert pk.pk_request_digest(other, d) == O.request_digest(other, d)


@pytest.mark.parametrize("field,value,code", [
    ("weight_precision", "auto", -3), ("kv_format", "", -3), ("model_id", "y" * 4097, -4),
])
def test_worker_digest_errors_match_oracle(pk, field, value, code):
    d = {"model_id": "m", "weight_precision": "bf16", "weight_version": "v", "kv_format": "bf16", field: value}
    with pytest.raises(pk.PKError) as e:
        pk.pk_worker_digest(d)
    assert e.value.code == code
    with pytest.raises(O.OracleError) as e2:
        O.worker_digest(d)
    assert e2.value.code == code


def test_request_digests_batch(pk):
    rng = np.random.default_rng(16)
    descs = [_rand_desc(rng) for _ in range(100)]
    w = bytes(rng.integers(0, 256, 32, dtype=np.uint8))
    got = pk.pk_request_digests(w, descs)
    for j, d in enumerate(descs):
        assert bytes(got[j]) == O.request_digest(w, d)


def test_request_digest_errors(pk):
    w = bytes(32)
    with pytest.raises(pk.PKError) as e:
        pk.pk_request_digest(w, {"salt": "s" * 4097})
    assert e.value.code == pk.PK_ERR_FIELD_TOO_LONG
    # the worker fields are not read by the request half: an unresolved dtype is not an error there
    assert pk.pk_request_digest(w, {"kv_format": "auto", "salt": "s"}) == O.request_digest(w, {"salt": "s"})


def test_content_identities_match_oracle(pk):
    rng = np.random.default_rng(21)
    for _ in range(200):
        top = bytes(rng.integers(0, 256, 32, dtype=np.uint8))
        shape = [int(x) for x in rng.integers(0, 5000, int(rng.integers(0, 5)))]
        name = bytes(rng.integers(0, 256, int(rng.integers(0, 40)), dtype=np.uint8))
        n = int(rng.integers(0, 1 << 40))
        t = pk.pk_tensor_identity(name, "bf16", shape, n, top)
        assert t == O.tensor_identity(name, "bf16", shape, n, top)
    ids = [bytes(rng.integers(0, 256, 32, dtype=np.uint8)) for _ in range(7)]
    cfg = ["r=8", "", "target_modules=q_proj,v_proj"]
    assert pk.pk_adapter_identity(ids, cfg) == O.adapter_identity(ids, cfg)
    assert pk.pk_adapter_identity([], []) == O.adapter_identity([], [])


def test_content_scratch_bytes(pk):
    assert pk.pk_content_scratch_bytes(0) == 32 and pk.pk_content_scratch_bytes(1024) == 32
    assert pk.pk_content_scratch_bytes(1025) == 2 * 32 + 32
    assert pk.pk_content_scratch_bytes(33 * 1024 + 1) == 34 * 32 + 2 * 32 + 32


def test_batch_encode_offsets(pk):
    rng = np.random.default_rng(6)
    descs = [_rand_desc(rng) for _ in range(64)]
    enc, off = pk.pk_descriptors_encode(descs)
    for j, d in enumerate(descs):
        assert bytes(enc[off[j]:off[j + 1]]) == O.enc(O.canonicalize(d))


@pytest.mark.parametrize("field,value,code", [
    ("weight_precision", "auto", -3), ("kv_format", "AUTO", -3), ("kv_format", "", -3),
    ("weight_precision", "", -3), ("salt", "x" * 4097, -4), ("model_id", "y" * 4097, -4),
])
def test_descriptor_errors_match_oracle(pk, field, value, code):
    d = {"model_id": "m", "weight_precision": "bf16", "weight_version": "v", "adapter_id": "", "kv_format": "bf16",
         "salt": ""}
    d[field] = value
    with pytest.raises(pk.PKError) as e:
        pk.pk_descriptor_digest(d)
    assert e.value.code == code
    with pytest.raises(O.OracleError) as e2:
        O.descriptor_digest(d)
    assert e2.value.code == code


def test_descriptor_field_limit_exact(pk):
    d = {"model_id": "m", "weight_precision": "bf16", "kv_format": "bf16", "salt": "s" * 4096}
    assert pk.pk_descriptor_digest(d) == O.descriptor_digest(d)


def test_table_bytes(pk):
    assert pk.pk_table_bytes(0) == 0 and pk.pk_table_bytes(32) == 0
    assert pk.pk_table_bytes(1) == 64 and pk.pk_table_bytes(20) == 32 << 20


def test_init_host_errors_before_any_cuda_call(pk):
    L = pk.lib()
    out = ctypes.c_void_p()
    # bad capacity and too-small table: rejected on the host (pointer never dereferenced)
    for log2, nbytes in ((0, 1 << 20), (32, 1 << 20), (10, 32 * 1024 - 1)):
        cfg = pk.pk_config(256, log2, 0, 4096, nbytes)
        assert L.pk_init(ctypes.byref(out), ctypes.byref(cfg), None) == pk.PK_ERR_CAPACITY
        assert out.value is None
    for cfg in (pk.pk_config(0, 10, 0, 4096, 1 << 20), pk.pk_config(256, 10, 0, 0, 1 << 20),
                pk.pk_config(256, 10, 0, 4100, 1 << 20)):
        assert L.pk_init(ctypes.byref(out), ctypes.byref(cfg), None) == pk.PK_ERR_ARG
    assert L.pk_init(None, ctypes.byref(pk.pk_config(256, 10, 0, 4096, 1 << 20)), None) == pk.PK_ERR_ARG


def test_null_context_rejected(pk):
    L = pk.lib()
    assert L.pk_lookup(None, None, None, 0, 0, None, None, None, None) == pk.PK_ERR_ARG
    assert L.pk_store(None, None, None, 0, None, None, 0, None, None, None, None) == pk.PK_ERR_ARG
    assert L.pk_lookup_store(None, None, None, None, 0, 0, None, None, None, None, None, None) == pk.PK_ERR_ARG
    assert L.pk_derive_keys(None, None, 0, None, 0, None, None, 0, None, None, 0, None, None) == pk.PK_ERR_ARG
    assert L.pk_destroy(None) == pk.PK_ERR_ARG


def test_key_string_and_model_tag_match_oracle(pk):
    rng = np.random.default_rng(21)
    for _ in range(300):
        p = rng.integers(0, 256, 16, dtype=np.uint8).tobytes()
        assert pk.pk_key_string(p) == O.key_string(p)
    for _ in range(50):
        d = _rand_desc(rng)
        try:
            want = O.model_tag(d)
        except O.OracleError as e:
            with pytest.raises(pk.PKError) as ei:
                pk.pk_model_tag(d)
            assert ei.value.code == e.code
            continue
        assert pk.pk_model_tag(d) == want


def test_key_strings_host_errors_before_any_cuda_call(pk):
    L = pk.lib()
    fake = ctypes.c_void_p(1 << 40)  # never dereferenced: every case fails its host check
    assert L.pk_key_strings(fake, 4, None, 0, 21, fake, None) == pk.PK_ERR_ARG           # width < 22
    assert L.pk_key_strings(fake, 4, None, 0, 257, fake, None) == pk.PK_ERR_ARG          # width > max
    assert L.pk_key_strings(fake, 4, b"abc", 3, 24, fake, None) == pk.PK_ERR_ARG         # prefix + 22 > width
    assert L.pk_key_strings(fake, 4, None, 2, 64, fake, None) == pk.PK_ERR_ARG           # prefix NULL
    assert L.pk_key_strings(None, 4, None, 0, 22, fake, None) == pk.PK_ERR_ARG           # keys NULL
    assert L.pk_key_strings(fake, 4, None, 0, 22, None, None) == pk.PK_ERR_ARG           # out NULL
    assert L.pk_key_strings(ctypes.c_void_p((1 << 40) + 8), 4, None, 0, 22, fake, None) == pk.PK_ERR_ARG
    assert L.pk_key_strings(fake, 4, None, 0, 22, ctypes.c_void_p((1 << 40) + 4), None) == pk.PK_ERR_ARG
    assert L.pk_key_strings(None, 0, None, 0, 22, None, None) == pk.PK_OK                # empty batch
