"""Pins of the oracle's two-level variant against what the paper fixes for it:
request-level (adapter, salt) and worker-level (precision, version, KV
representation, with the model identity) provenance bound through separate
digests (Sec. 2.2), the worker half taken over resolved values, the
request-level binding inert for a request with neither adapter nor salt, and
the two halves composing independently (Sec. 5.3), with the contract's key-level
properties (Def. 2, Eq. 4).  The byte layout of the halves is this build's
reading and is not pinned by the paper (no worked values are printed)."""
import itertools

import numpy as np
import pytest

import oracle as O

BASE = {"model_id": "synthetic/model-7b", "weight_precision": "bf16", "weight_version": "0123abcd",
        "adapter_id": "", "kv_format": "fp8_e4m3", "salt": ""}


def keys_of(tokens, C, d):
    return O.request_keys(np.asarray(tokens, np.int32), C, d)


def test_inert_request_keys_as_the_worker_only_chain():
    rng = np.random.default_rng(1)
    toks = rng.integers(0, 152064, 4 * 256).astype(np.int32)
    w = O.worker_digest(BASE)
    assert O.request_digest(w, BASE) == w                      # the binding is inert ...
    assert np.array_equal(keys_of(toks, 256, O.request_digest(w, BASE)), keys_of(toks, 256, w))  # ... key for key
    for other in (dict(BASE, adapter_id="adapter-00"), dict(BASE, salt="t"), dict(BASE, extra=[b""])):
        assert O.request_digest(w, other) != w                 # any request-level tag binds


def test_worker_half_ignores_request_fields_and_request_half_ignores_worker_fields():
    w = O.worker_digest(BASE)
    for f, v in (("adapter_id", "a"), ("salt", "s")):
        assert O.worker_digest(dict(BASE, **{f: v})) == w
    assert O.worker_digest(dict(BASE, extra=[b"x"])) == w
    q = dict(BASE, adapter_id="adapter-03", salt="tenant")
    for f, v in (("model_id", "other"), ("weight_precision", "fp16"), ("weight_version", "ff"), ("kv_format", "bf16")):
        changed = dict(q, **{f: v})
        assert O.request_half(changed) == O.request_half(q)
        assert O.worker_digest(changed) != w                    # separate digests: only the worker half moves


@pytest.mark.parametrize("field,value", [("model_id", "synthetic/model-7b-v2"), ("weight_precision", "fp8_e4m3"),
                                         ("weight_version", "0123abce"), ("kv_format", "fp8_e5m2"),
                                         ("adapter_id", "adapter-01"), ("salt", "tenant-b")])
def test_differential_omission_every_dimension_changes_every_key(field, value):
    """Eq. 4: changing one registered dimension changes every key of a request,
    for inert and tagged requests alike."""
    rng = np.random.default_rng(2)
    toks = rng.integers(0, 32000, 6 * 64).astype(np.int32)
    for base in (BASE, dict(BASE, adapter_id="adapter-00", salt="tenant-a")):
        a = keys_of(toks, 64, O.request_digest(O.worker_digest(base), base))
        other = dict(base, **{field: value})
        b = keys_of(toks, 64, O.request_digest(O.worker_digest(other), other))
        assert not np.any(np.all(a == b, axis=1))


def test_grid_of_provenance_classes_gives_distinct_digests():
    """Every combination of the five dimensions (and inert vs tagged) maps to its
    own digest: no two provenance classes merge (Def. 2)."""
    grid = {"weight_precision": ["bf16", "fp8_e4m3"], "weight_version": ["v1", "v2"], "kv_format": ["bf16", "fp16"],
            "adapter_id": ["", "adapter-00", "adapter-01"], "salt": ["", "a", "b"]}
    seen = {}
    for combo in itertools.product(*grid.values()):
        d = dict(BASE, **dict(zip(grid, combo)))
        dg = O.request_digest(O.worker_digest(d), d)
        assert dg not in seen, (combo, seen.get(dg))
        seen[dg] = combo
    assert len(seen) == 2 * 2 * 2 * 3 * 3


def test_field_boundaries_and_tag_positions_are_distinct():
    w = O.worker_digest(BASE)
    pairs = [({"adapter_id": "ab", "salt": "c"}, {"adapter_id": "a", "salt": "bc"}),
             ({"adapter_id": "x"}, {"salt": "x"}),
             ({"salt": "x"}, {"extra": [b"x"]}),
             ({"extra": [b""]}, {"extra": [b"", b""]})]
    for a, b in pairs:
        assert O.request_digest(w, dict(BASE, **a)) != O.request_digest(w, dict(BASE, **b)), (a, b)


def test_worker_half_is_canonical_and_refuses_unresolved_values():
    assert O.worker_digest(dict(BASE, weight_precision="BFloat16")) == O.worker_digest(BASE)
    assert O.worker_digest(dict(BASE, kv_format="FLOAT8_E4M3FN")) == O.worker_digest(BASE)
    assert O.worker_digest(dict(BASE, kv_format="fp8")) != O.worker_digest(BASE)   # distinct formats never merge
    for f in ("weight_precision", "kv_format"):
        with pytest.raises(O.OracleError) as e:
            O.worker_digest(dict(BASE, **{f: "auto"}))
        assert e.value.code == O.PK_ERR_UNRESOLVED


def test_request_digest_is_a_function_of_the_worker_digest_and_the_tags():
    """Cross-worker stability (Sec. 5.1): two workers with the same resolved
    values and a request with the same tags derive the same digest."""
    a = dict(BASE, adapter_id="adapter-05", salt="t")
    b = {"model_id": BASE["model_id"], "weight_precision": "BF16", "weight_version": BASE["weight_version"],
         "kv_format": "float8_e4m3fn", "adapter_id": "adapter-05", "salt": "t"}
    assert O.request_digest(O.worker_digest(a), a) == O.request_digest(O.worker_digest(b), b)
