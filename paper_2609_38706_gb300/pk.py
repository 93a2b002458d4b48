"""Thin Python binding of libpk (include/pk.h).

Argument marshalling only: every function has the name of the C entry point
it calls, turns tensors into raw pointers and sizes, passes the CUDA stream
handle, and raises ``PKError`` on a negative status.  All computation happens
in the library's CUDA kernels (and its host canonicaliser); there is no
fallback: if ``libpk.so`` has not been built this module raises on first use.
"""
from __future__ import annotations

import ctypes
import os
from typing import Iterable, Mapping, Optional, Sequence

import numpy as np
import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build", "libpk.so")

PK_OK = 0
PK_ERR_ARG = -1
PK_ERR_CAPACITY = -2
PK_ERR_UNRESOLVED = -3
PK_ERR_FIELD_TOO_LONG = -4
PK_ERR_TABLE_FULL = -5
PK_ERR_PROBE_LIMIT = -6
PK_ERR_RESERVED_KEY = -7
PK_ERR_CUDA = -8
PK_ERR_TOO_LARGE = -9
PK_ERR_TIMEOUT = -10
PK_PAGE_ABSENT, PK_PAGE_EQUAL, PK_PAGE_DIFFERS = 0, 1, 2
PK_NOALLOC_MAX_ENTRIES = 1 << 18
PK_STORE_SKIPPED = 0
PK_STORE_INSERTED = 1
PK_STORE_PRESENT = 2
PK_NO_SLOT = 0xFFFFFFFF
PK_KEY_BYTES = 32
PK_ENTRY_BYTES = 32
PK_KEY_STRING_CHARS = 22
PK_KEY_STRING_MAX_WIDTH = 256
REGISTRY_V1 = ("model_id", "weight_precision", "weight_version", "adapter_id", "kv_format", "salt")


class PKError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {pk_strerror(code)} ({code})")
        self.code = code


class pk_bytes(ctypes.Structure):
    _fields_ = [("p", ctypes.c_void_p), ("len", ctypes.c_uint32)]


class pk_descriptor(ctypes.Structure):
    _fields_ = [(name, pk_bytes) for name in REGISTRY_V1] + [
        ("extra", ctypes.POINTER(pk_bytes)), ("n_extra", ctypes.c_uint32)]


class pk_config(ctypes.Structure):
    _fields_ = [("chunk_tokens", ctypes.c_uint32), ("capacity_log2", ctypes.c_uint32),
                ("max_probe", ctypes.c_uint32), ("table_dev", ctypes.c_void_p),
                ("table_bytes", ctypes.c_size_t)]


_lib = None
_VP, _U32, _U64, _I32 = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int32


def lib() -> ctypes.CDLL:
    """Load libpk.so (built by ``__graft_entry__.build()``); raise if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"libpk.so not found at {_LIB_PATH}: build it first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(_LIB_PATH)
        sig = {
            "pk_table_bytes": (ctypes.c_size_t, [_U32]),
            "pk_init": (ctypes.c_int, [ctypes.POINTER(_VP), ctypes.POINTER(pk_config), _VP]),
            "pk_destroy": (ctypes.c_int, [_VP]),
            "pk_descriptor_encode": (ctypes.c_int, [ctypes.POINTER(pk_descriptor), _VP, ctypes.c_size_t,
                                                    ctypes.POINTER(ctypes.c_size_t)]),
            "pk_descriptors_encode": (ctypes.c_int, [ctypes.POINTER(pk_descriptor), _U32, _VP,
                                                     ctypes.c_size_t, _VP]),
            "pk_descriptor_digest": (ctypes.c_int, [ctypes.POINTER(pk_descriptor), _VP]),
            "pk_worker_digest": (ctypes.c_int, [ctypes.POINTER(pk_descriptor), _VP]),
            "pk_request_digest": (ctypes.c_int, [_VP, ctypes.POINTER(pk_descriptor), _VP]),
            "pk_request_digests": (ctypes.c_int, [_VP, ctypes.POINTER(pk_descriptor), _U32, _VP]),
            "pk_digest_descriptors": (ctypes.c_int, [_VP, _VP, _U64, _VP, _U32, _VP, _VP, _VP]),
            "pk_derive_keys": (ctypes.c_int, [_VP, _VP, _U64, _VP, _U32, _VP, _VP, _U32, _VP, _VP, _U64,
                                              _VP, _VP]),
            "pk_derive_keys_enc": (ctypes.c_int, [_VP, _VP, _U64, _VP, _U32, _VP, _VP, _U64, _VP, _U32, _VP, _VP, _VP,
                                                  _U64, _VP, _VP]),
            "pk_lookup": (ctypes.c_int, [_VP, _VP, _VP, _U32, _U64, _VP, _VP, _VP, _VP]),
            "pk_store": (ctypes.c_int, [_VP, _VP, _VP, _U64, _VP, _VP, _U32, _VP, _VP, _VP, _VP]),
            "pk_lookup_store": (ctypes.c_int, [_VP, _VP, _VP, _VP, _U32, _U64, _VP, _VP, _VP, _VP, _VP, _VP]),
            "pk_derive_lookup_store": (ctypes.c_int, [_VP, _VP, _U64, _VP, _U32, _VP, _VP, _U64, _VP, _U32, _VP, _VP,
                                                      _VP, _U64, _VP, _VP, _VP, _VP, _VP, _VP, _VP]),
            "pk_entries": (ctypes.c_int, [_VP, ctypes.POINTER(ctypes.c_uint64), _VP]),
            "pk_store_noalloc": (ctypes.c_int, [ctypes.POINTER(pk_config), _VP, _VP, _U64, _VP, _VP, _U32, _VP, _VP,
                                                _VP, _VP]),
            "pk_compare_pages": (ctypes.c_int, [_VP, _VP, _VP, _U64, _U64, _U64, _VP, _VP, _VP, _VP]),
            "pk_content_scratch_bytes": (ctypes.c_size_t, [_U64]),
            "pk_content_digest": (ctypes.c_int, [_VP, _U64, _VP, ctypes.c_size_t, _VP, _VP]),
            "pk_content_scratch_bytes_batch": (ctypes.c_size_t, [_VP, _U32]),
            "pk_content_digests": (ctypes.c_int, [_VP, _VP, _U32, _VP, ctypes.c_size_t, _VP, _VP]),
            "pk_tensor_identity": (ctypes.c_int, [ctypes.POINTER(pk_bytes), ctypes.POINTER(pk_bytes), _VP, _U32,
                                                  _U64, _VP, _VP]),
            "pk_adapter_identity": (ctypes.c_int, [_VP, _U32, ctypes.POINTER(pk_bytes), _U32, _VP]),
            "pk_stamps_bytes": (ctypes.c_size_t, [_U32]),
            "pk_attach_stamps": (ctypes.c_int, [_VP, _VP, ctypes.c_size_t, _VP]),
            "pk_evict_scratch_bytes": (ctypes.c_size_t, [_U32]),
            "pk_evict": (ctypes.c_int, [_VP, _U64, _U64, _VP, ctypes.c_size_t, _VP, _U64, _VP, _VP, _VP]),
            "pk_evict_barrier_timeout_test": (ctypes.c_int, [_VP, _U64, _VP, ctypes.c_size_t, _U32, _VP, _VP]),
            "pk_key_string": (ctypes.c_int, [_VP, _VP]),
            "pk_model_tag": (ctypes.c_int, [ctypes.POINTER(pk_descriptor), _VP]),
            "pk_key_strings": (ctypes.c_int, [_VP, _U64, _VP, _U32, _U32, _VP, _VP]),
            "pk_table_save": (ctypes.c_int, [_VP, _VP, ctypes.c_size_t, _VP]),
            "pk_table_load": (ctypes.c_int, [_VP, _VP, ctypes.c_size_t, _VP]),
            "pk_strerror": (ctypes.c_char_p, [ctypes.c_int]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype, f.argtypes = res, args
        _lib = L
    return _lib


def _check(rc: int, where: str) -> None:
    if rc != PK_OK:
        raise PKError(rc, where)


def _p(t) -> Optional[int]:
    """Raw pointer of a tensor / ndarray (None for None)."""
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        return t.data_ptr() if t.numel() else None
    if isinstance(t, np.ndarray):
        return t.ctypes.data if t.size else None
    return int(t)


def _s(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else None
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


class Descriptors:
    """ctypes array of pk_descriptor built from dicts (field name -> str/bytes,
    optional ``extra`` list), keeping the byte buffers alive."""

    def __init__(self, descs: Iterable[Mapping]):
        descs = list(descs)
        self._keep = []
        self.array = (pk_descriptor * max(len(descs), 1))()
        self.count = len(descs)
        for j, d in enumerate(descs):
            for name in REGISTRY_V1:
                setattr(self.array[j], name, self._b(d.get(name, b"")))
            extra = list(d.get("extra", ()) or ())
            if extra:
                arr = (pk_bytes * len(extra))(*[self._b(x) for x in extra])
                self._keep.append(arr)
                self.array[j].extra = ctypes.cast(arr, ctypes.POINTER(pk_bytes))
                self.array[j].n_extra = len(extra)

    def _b(self, v) -> pk_bytes:
        if v is None:
            v = b""
        if isinstance(v, str):
            v = v.encode("utf-8")
        v = bytes(v)
        buf = ctypes.create_string_buffer(v, len(v) + 1)
        self._keep.append(buf)
        return pk_bytes(ctypes.cast(buf, ctypes.c_void_p), len(v))


def _descs(d) -> Descriptors:
    return d if isinstance(d, Descriptors) else Descriptors(d)


# ---------------------------------------------------------------------------
# entry points
# ---------------------------------------------------------------------------
def pk_strerror(code: int) -> str:
    try:
        return lib().pk_strerror(code).decode()
    except RuntimeError:
        return f"status {code}"


def pk_table_bytes(capacity_log2: int) -> int:
    return int(lib().pk_table_bytes(capacity_log2))


def pk_init(table: torch.Tensor, chunk_tokens: int, capacity_log2: int, max_probe: int = 0,
            stream=None) -> int:
    """Bind a caller-owned table tensor (>= pk_table_bytes bytes) and clear it.
    Returns the opaque context pointer."""
    cfg = pk_config(chunk_tokens, capacity_log2, max_probe, _p(table),
                    table.numel() * table.element_size())
    out = ctypes.c_void_p()
    _check(lib().pk_init(ctypes.byref(out), ctypes.byref(cfg), _s(stream)), "pk_init")
    return out.value


def pk_destroy(ctx: int) -> None:
    _check(lib().pk_destroy(ctx), "pk_destroy")


def pk_descriptor_encode(desc) -> bytes:
    d = _descs([desc]) if isinstance(desc, Mapping) else _descs(desc)
    n = ctypes.c_size_t(0)
    rc = lib().pk_descriptor_encode(d.array, None, 0, ctypes.byref(n))
    if rc not in (PK_OK, PK_ERR_ARG):
        _check(rc, "pk_descriptor_encode")
    buf = ctypes.create_string_buffer(max(n.value, 1))
    _check(lib().pk_descriptor_encode(d.array, buf, n.value, ctypes.byref(n)), "pk_descriptor_encode")
    return buf.raw[: n.value]


def pk_descriptors_encode(descs, out: Optional[np.ndarray] = None,
                          enc_off: Optional[np.ndarray] = None) -> tuple[np.ndarray, np.ndarray]:
    """Encode D descriptors into ``out`` (uint8, host; pinned tensors welcome)
    and ``enc_off`` (int64[D+1]).  Returns views (bytes used, offsets)."""
    d = _descs(descs)
    if out is None:
        out = np.zeros(64 * 1024 + d.count * (7 * 4 + 8 * 4096), np.uint8)
    if enc_off is None:
        enc_off = np.zeros(d.count + 1, np.int64)
    cap = out.numel() if isinstance(out, torch.Tensor) else out.size
    _check(lib().pk_descriptors_encode(d.array, d.count, _p(out), cap, _p(enc_off)), "pk_descriptors_encode")
    used = int(enc_off[d.count])
    return out[:used], enc_off


def pk_descriptor_digest(desc) -> bytes:
    d = _descs([desc]) if isinstance(desc, Mapping) else _descs(desc)
    out = (ctypes.c_uint8 * 32)()
    _check(lib().pk_descriptor_digest(d.array, out), "pk_descriptor_digest")
    return bytes(out)


def pk_worker_digest(desc) -> bytes:
    d = _descs([desc]) if isinstance(desc, Mapping) else _descs(desc)
    out = (ctypes.c_uint8 * 32)()
    _check(lib().pk_worker_digest(d.array, out), "pk_worker_digest")
    return bytes(out)


def pk_request_digest(worker: bytes, desc) -> bytes:
    d = _descs([desc]) if isinstance(desc, Mapping) else _descs(desc)
    w = (ctypes.c_uint8 * 32).from_buffer_copy(bytes(worker))
    out = (ctypes.c_uint8 * 32)()
    _check(lib().pk_request_digest(w, d.array, out), "pk_request_digest")
    return bytes(out)


def pk_request_digests(worker: bytes, descs) -> np.ndarray:
    """uint8[n][32]: pk_request_digest of each descriptor under one worker digest."""
    d = _descs(descs)
    w = (ctypes.c_uint8 * 32).from_buffer_copy(bytes(worker))
    out = np.zeros((max(d.count, 1), 32), np.uint8)
    _check(lib().pk_request_digests(w, d.array, d.count, _p(out)), "pk_request_digests")
    return out[: d.count]


def two_level_digests(descs) -> np.ndarray:
    """uint8[D][32]: the two-level digest of each descriptor (its own worker
    half, then its request half)."""
    out = np.zeros((len(descs), 32), np.uint8)
    for j, d in enumerate(descs):
        out[j] = np.frombuffer(pk_request_digest(pk_worker_digest(d), d), np.uint8)
    return out


def pk_digest_descriptors(ctx: int, enc: torch.Tensor, enc_off: torch.Tensor, digests: torch.Tensor,
                          status: torch.Tensor, stream=None) -> None:
    D = enc_off.numel() - 1
    _check(lib().pk_digest_descriptors(ctx, _p(enc), enc.numel(), _p(enc_off), D, _p(digests), _p(status),
                                       _s(stream)), "pk_digest_descriptors")


def pk_derive_keys(ctx: int, tokens: torch.Tensor, tok_off: torch.Tensor, desc_idx: torch.Tensor,
                   digests: torch.Tensor, key_off: torch.Tensor, keys: torch.Tensor, status: torch.Tensor,
                   stream=None) -> None:
    R = tok_off.numel() - 1
    D = digests.numel() // 32
    _check(lib().pk_derive_keys(ctx, _p(tokens), tokens.numel(), _p(tok_off), R, _p(desc_idx), _p(digests), D,
                                _p(key_off), _p(keys), keys.numel() // 32, _p(status), _s(stream)),
           "pk_derive_keys")


def pk_derive_keys_enc(ctx: int, tokens: torch.Tensor, tok_off: torch.Tensor, desc_idx: torch.Tensor,
                       enc: torch.Tensor, enc_off: torch.Tensor, digests: torch.Tensor, key_off: torch.Tensor,
                       keys: torch.Tensor, status: torch.Tensor, stream=None) -> None:
    R = tok_off.numel() - 1
    D = enc_off.numel() - 1
    _check(lib().pk_derive_keys_enc(ctx, _p(tokens), tokens.numel(), _p(tok_off), R, _p(desc_idx), _p(enc),
                                    enc.numel(), _p(enc_off), D, _p(digests), _p(key_off), _p(keys),
                                    keys.numel() // 32, _p(status), _s(stream)), "pk_derive_keys_enc")


def pk_lookup(ctx: int, keys: torch.Tensor, key_off: torch.Tensor, hit_chunks: torch.Tensor,
              slots: torch.Tensor, status: torch.Tensor, stream=None) -> None:
    R = key_off.numel() - 1
    _check(lib().pk_lookup(ctx, _p(keys), _p(key_off), R, keys.numel() // 32, _p(hit_chunks), _p(slots),
                           _p(status), _s(stream)), "pk_lookup")


def pk_store(ctx: int, keys: torch.Tensor, slots: torch.Tensor, result: torch.Tensor, slot_out: torch.Tensor,
             status: torch.Tensor, key_off: Optional[torch.Tensor] = None,
             hit_chunks: Optional[torch.Tensor] = None, stream=None) -> None:
    n = keys.numel() // 32
    R = 0 if key_off is None else key_off.numel() - 1
    _check(lib().pk_store(ctx, _p(keys), _p(slots), n, _p(key_off), _p(hit_chunks), R, _p(result), _p(slot_out),
                          _p(status), _s(stream)), "pk_store")


def pk_lookup_store(ctx: int, keys: torch.Tensor, new_slots: torch.Tensor, key_off: torch.Tensor,
                    hit_chunks: torch.Tensor, slots: torch.Tensor, result: torch.Tensor, slot_out: torch.Tensor,
                    status: torch.Tensor, stream=None) -> None:
    R = key_off.numel() - 1
    _check(lib().pk_lookup_store(ctx, _p(keys), _p(new_slots), _p(key_off), R, keys.numel() // 32,
                                 _p(hit_chunks), _p(slots), _p(result), _p(slot_out), _p(status), _s(stream)),
           "pk_lookup_store")


def pk_derive_lookup_store(ctx: int, tokens: torch.Tensor, tok_off: torch.Tensor, desc_idx: torch.Tensor,
                           enc: torch.Tensor, enc_off: torch.Tensor, digests: torch.Tensor, key_off: torch.Tensor,
                           keys: torch.Tensor, new_slots: torch.Tensor, hit_chunks: torch.Tensor, slots: torch.Tensor,
                           result: torch.Tensor, slot_out: torch.Tensor, status: torch.Tensor, stream=None) -> None:
    R = tok_off.numel() - 1
    D = enc_off.numel() - 1
    _check(lib().pk_derive_lookup_store(ctx, _p(tokens), tokens.numel(), _p(tok_off), R, _p(desc_idx), _p(enc),
                                        enc.numel(), _p(enc_off), D, _p(digests), _p(key_off), _p(keys),
                                        keys.numel() // 32, _p(new_slots), _p(hit_chunks), _p(slots), _p(result),
                                        _p(slot_out), _p(status), _s(stream)), "pk_derive_lookup_store")


def pk_compare_pages(slots: torch.Tensor, pages: torch.Tensor, ref_pages: torch.Tensor, verdict: torch.Tensor,
                     counts: torch.Tensor, status: torch.Tensor, stream=None) -> None:
    """pages: uint8 [n, page_bytes]; ref_pages: uint8 [n_ref, page_bytes]; counts: int64[3] (accumulated)."""
    n, page_bytes = pages.shape
    _check(lib().pk_compare_pages(_p(slots), _p(pages), _p(ref_pages), n, ref_pages.shape[0], page_bytes,
                                  _p(verdict), _p(counts), _p(status), _s(stream)), "pk_compare_pages")


def pk_content_scratch_bytes(n_bytes: int) -> int:
    return int(lib().pk_content_scratch_bytes(n_bytes))


def pk_content_digest(data: torch.Tensor, scratch: torch.Tensor, top: torch.Tensor, stream=None) -> None:
    """top (uint8[32], device) = tree top of the bytes of `data` (a contiguous device tensor)."""
    n = data.numel() * data.element_size()
    _check(lib().pk_content_digest(_p(data), n, _p(scratch), scratch.numel(), _p(top), _s(stream)),
           "pk_content_digest")


def pk_content_scratch_bytes_batch(sizes) -> int:
    arr = (ctypes.c_uint64 * max(len(sizes), 1))(*[int(x) for x in sizes])
    return int(lib().pk_content_scratch_bytes_batch(arr, len(sizes)))


def pk_content_digests(datas, scratch: torch.Tensor, tops: torch.Tensor, stream=None) -> None:
    """tops (uint8[n, 32], device) = the tree tops of the contiguous device tensors `datas`."""
    n = len(datas)
    ptrs = (ctypes.c_void_p * max(n, 1))(*[_p(d) for d in datas])
    sizes = (ctypes.c_uint64 * max(n, 1))(*[d.numel() * d.element_size() for d in datas])
    _check(lib().pk_content_digests(ptrs, sizes, n, _p(scratch), scratch.numel(), _p(tops), _s(stream)),
           "pk_content_digests")


def _pkb(b: bytes):
    buf = ctypes.create_string_buffer(bytes(b), max(len(b), 1))
    return pk_bytes(ctypes.cast(buf, ctypes.c_void_p), len(b)), buf


def pk_tensor_identity(name, dtype, shape, n_bytes: int, top: bytes) -> bytes:
    nb, k1 = _pkb(name.encode() if isinstance(name, str) else name)
    db, k2 = _pkb(dtype.encode() if isinstance(dtype, str) else dtype)
    dims = (ctypes.c_int64 * max(len(shape), 1))(*[int(x) for x in shape])
    t = (ctypes.c_uint8 * 32).from_buffer_copy(bytes(top))
    out = (ctypes.c_uint8 * 32)()
    _check(lib().pk_tensor_identity(ctypes.byref(nb), ctypes.byref(db), dims, len(shape), n_bytes, t, out),
           "pk_tensor_identity")
    return bytes(out)


def pk_adapter_identity(tensor_ids, config) -> bytes:
    ids = np.frombuffer(b"".join(bytes(x) for x in tensor_ids), np.uint8) if tensor_ids else np.zeros(32, np.uint8)
    keep = [_pkb(c.encode() if isinstance(c, str) else c) for c in config]
    arr = (pk_bytes * max(len(keep), 1))(*[k[0] for k in keep])
    out = (ctypes.c_uint8 * 32)()
    _check(lib().pk_adapter_identity(ids.ctypes.data, len(tensor_ids), arr, len(keep), out), "pk_adapter_identity")
    return bytes(out)


def pk_stamps_bytes(capacity_log2: int) -> int:
    return int(lib().pk_stamps_bytes(capacity_log2))


def pk_attach_stamps(ctx: int, stamps: Optional[torch.Tensor], stream=None) -> None:
    """Budget mode on (stamps: device buffer of pk_stamps_bytes, zeroed here) or off (None)."""
    nbytes = 0 if stamps is None else stamps.numel() * stamps.element_size()
    _check(lib().pk_attach_stamps(ctx, _p(stamps), nbytes, _s(stream)), "pk_attach_stamps")


def pk_evict_scratch_bytes(capacity_log2: int) -> int:
    return int(lib().pk_evict_scratch_bytes(capacity_log2))


def pk_evict(ctx: int, budget: int, keep: int, scratch: torch.Tensor, evicted: Optional[torch.Tensor],
             n_evicted: Optional[torch.Tensor], status: torch.Tensor, stream=None) -> None:
    """evicted: uint32/int32 [cap] device (or None); n_evicted: int64[1] device (or None)."""
    _check(lib().pk_evict(ctx, budget, keep, _p(scratch), scratch.numel(), _p(evicted),
                          0 if evicted is None else evicted.numel(), _p(n_evicted), _p(status), _s(stream)),
           "pk_evict")


def pk_evict_barrier_timeout_test(ctx: int, budget: int, scratch: torch.Tensor, spin_limit: int,
                                  status: torch.Tensor, stream=None) -> None:
    """Test hook: pk_evict with CTA 0 withholding its first barrier arrival and
    the waits bounded at spin_limit polls (the status must end PK_ERR_TIMEOUT)."""
    _check(lib().pk_evict_barrier_timeout_test(ctx, budget, _p(scratch), scratch.numel(), spin_limit, _p(status),
                                               _s(stream)), "pk_evict_barrier_timeout_test")


def pk_key_string(key16: bytes) -> str:
    """The 22 base64 characters of a 16-byte key prefix (host)."""
    if len(bytes(key16)) != 16:
        raise PKError(PK_ERR_ARG, "pk_key_string")
    k = (ctypes.c_uint8 * 16).from_buffer_copy(bytes(key16))
    out = (ctypes.c_char * 22)()
    _check(lib().pk_key_string(k, out), "pk_key_string")
    return out.raw.decode("ascii")


def pk_model_tag(desc) -> str:
    """The 22-character hash of the model identity and worker provenance (host)."""
    d = _descs([desc]) if isinstance(desc, Mapping) else _descs(desc)
    out = (ctypes.c_char * 22)()
    _check(lib().pk_model_tag(d.array, out), "pk_model_tag")
    return out.raw.decode("ascii")


def pk_key_strings(keys: torch.Tensor, prefix: bytes, width: int, out: torch.Tensor, n: Optional[int] = None,
                   stream=None) -> None:
    """out (uint8 [n, width], device): row i = prefix || base64 of keys[i, :16] || zero fill."""
    n = keys.shape[0] if n is None else n
    pre = bytes(prefix)
    buf = ctypes.create_string_buffer(pre, max(len(pre), 1))
    _check(lib().pk_key_strings(_p(keys), n, ctypes.cast(buf, ctypes.c_void_p), len(pre), width, _p(out),
                                _s(stream)), "pk_key_strings")


def pk_table_save(ctx: int, dst: torch.Tensor, stream=None) -> None:
    _check(lib().pk_table_save(ctx, _p(dst), dst.numel() * dst.element_size(), _s(stream)), "pk_table_save")


def pk_table_load(ctx: int, src: torch.Tensor, stream=None) -> None:
    _check(lib().pk_table_load(ctx, _p(src), src.numel() * src.element_size(), _s(stream)), "pk_table_load")


def pk_store_noalloc(table: torch.Tensor, capacity_log2: int, keys: torch.Tensor, slots: torch.Tensor,
                     result: torch.Tensor, slot_out: torch.Tensor, status: torch.Tensor, max_probe: int = 0,
                     key_off: Optional[torch.Tensor] = None, hit_chunks: Optional[torch.Tensor] = None,
                     stream=None) -> None:
    """pk_store without a context, for callers that cannot allocate device
    memory; the table tensor must be zero-filled before its first use."""
    cfg = pk_config(1, capacity_log2, max_probe, _p(table), table.numel() * table.element_size())
    n = keys.numel() // 32
    R = 0 if key_off is None else key_off.numel() - 1
    _check(lib().pk_store_noalloc(ctypes.byref(cfg), _p(keys), _p(slots), n, _p(key_off), _p(hit_chunks), R,
                                  _p(result), _p(slot_out), _p(status), _s(stream)), "pk_store_noalloc")


def pk_entries(ctx: int, stream=None) -> int:
    v = ctypes.c_uint64(0)
    _check(lib().pk_entries(ctx, ctypes.byref(v), _s(stream)), "pk_entries")
    return int(v.value)
