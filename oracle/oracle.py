"""CPU oracle for provenance-bound KV-cache keys -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference leg
of ``bench.py`` may import this module.  It shares no code with the CUDA path
(``paper_2609_38706_gb300``) and imports nothing from it.

Every function restates one passage of the paper ("Preserving Provenance in
Shared KV Caches for LLM Serving") or one of the stated readings where the
paper is silent:

* ``canonicalize``   -- Sec. 5.3 "Worker-level digest": bind resolved values,
  never a launch string such as ``auto``; identity functions must be injective
  and cross-worker stable (Sec. 5.1).  The synonym table is a reading.
* ``enc``            -- Sec. 5.2, Eq. 3: an injective, length-prefixed encoder.
  Byte layout is a reading: LE32(field count) then LE32(len) || bytes per field.
* ``descriptor_digest`` -- d = H(enc(...)) of Eq. 3 with H = SHA-256.
* ``chunk_digest`` / ``chain_step`` / ``derive_keys`` -- the connector key f of
  Eq. 3 instantiated as c_i = SHA-256(LE int32 tokens of chunk i) and
  k_i = SHA-256(k_{i-1} || d || c_i) with k_{-1} = 0^32, full chunks only
  (Sec. 4.4: prefixes below one chunk never collide).  Computed by the plain C
  library ``pk_oracle.c`` (FIPS 180-4 written out).
* ``DictTable``      -- the shared store of Sec. 2.1 reduced to a map from the
  128-bit key prefix (Sec. 5.3, "the encoding keeps 128 bits") to a chunk
  slot.  Lookup returns the longest all-hit prefix (Sec. 2.1: on a local miss
  the connector queries the store; a hit skips that prefill, a miss computes
  and writes new state).  Store inserts in array order, the first occurrence
  wins, an existing key keeps its slot.
* ``SortedTable``    -- the same semantics computed with sort / searchsorted so
  that million-entry tables stay tractable; checked against ``DictTable``.

Pins live in ``tests/test_oracle_*.py``: SHA-256 against hashlib and the
FIPS 180-2 Appendix B digests, ``enc`` injectivity by property tests, the key
chain against the contract invariants Eq. 1, Eq. 2 and Eq. 4 by brute force,
and the tables against each other and against closed-form counts.  Parity
unpinned by the paper (stated conventions only): the field order of ``enc``,
its byte layout, the chain's operand order and zero seed, the partial-chunk
rule, which 16 bytes form the prefix, and the canonical synonym spellings.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Iterable, Mapping, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pk_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "libpk_oracle.so")

# Status vocabulary (the C-ABI's published codes, restated here as plain data).
PK_OK = 0
PK_ERR_ARG = -1
PK_ERR_CAPACITY = -2
PK_ERR_UNRESOLVED = -3
PK_ERR_FIELD_TOO_LONG = -4
PK_ERR_TABLE_FULL = -5
PK_ERR_PROBE_LIMIT = -6
PK_ERR_RESERVED_KEY = -7

STORE_SKIPPED = 0
STORE_INSERTED = 1
STORE_PRESENT = 2
NO_SLOT = 0xFFFFFFFF

MAX_FIELD_BYTES = 4096

# Registry v1 (Sec. 5.1 dimensions plus the model identity the connector already
# carries, Sec. 5.3).  Order is a stated convention.
REGISTRY_V1 = ("model_id", "weight_precision", "weight_version", "adapter_id", "kv_format", "salt")
_RESOLVED_FIELDS = ("weight_precision", "kv_format")
_SYNONYMS = {
    "bfloat16": "bf16",
    "float16": "fp16",
    "half": "fp16",
    "float32": "fp32",
    "float": "fp32",
    "float8_e4m3fn": "fp8_e4m3",
    "float8_e5m2": "fp8_e5m2",
}


class OracleError(Exception):
    def __init__(self, code: int, msg: str = ""):
        super().__init__(f"{code}: {msg}")
        self.code = code


# --------------------------------------------------------------------------
# C library
# --------------------------------------------------------------------------
_lib = None
_lib_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile pk_oracle.c with gcc into oracle/_build/libpk_oracle.so."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-o", tmp, _SRC])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lib_lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB_PATH)
            u8p = ctypes.POINTER(ctypes.c_uint8)
            L.oracle_sha256.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_void_p]
            L.oracle_sha256.restype = None
            L.oracle_chunk_digest.argtypes = [ctypes.c_void_p, ctypes.c_uint32, ctypes.c_void_p]
            L.oracle_chunk_digest.restype = None
            L.oracle_chain_step.argtypes = [ctypes.c_void_p] * 4
            L.oracle_chain_step.restype = None
            L.oracle_request_keys.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint32,
                                              ctypes.c_void_p, ctypes.c_void_p]
            L.oracle_request_keys.restype = ctypes.c_uint64
            L.oracle_derive_keys.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint32,
                                             ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p,
                                             ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p]
            L.oracle_derive_keys.restype = ctypes.c_int64
            L.oracle_max_threads.argtypes = []
            L.oracle_max_threads.restype = ctypes.c_int
            L.oracle_set_threads.argtypes = [ctypes.c_int]
            L.oracle_set_threads.restype = None
            L.oracle_constants.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
            L.oracle_constants.restype = None
            del u8p
            _lib = L
    return _lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def max_threads() -> int:
    return int(lib().oracle_max_threads())


def set_threads(n: int) -> None:
    lib().oracle_set_threads(int(n))


def constants() -> tuple[np.ndarray, np.ndarray]:
    k = np.zeros(64, np.uint32)
    h = np.zeros(8, np.uint32)
    lib().oracle_constants(_ptr(k), _ptr(h))
    return k, h


# --------------------------------------------------------------------------
# SHA-256 and the key chain
# --------------------------------------------------------------------------
def sha256(msg: bytes) -> bytes:
    buf = np.frombuffer(bytes(msg) + b"\0", dtype=np.uint8)
    out = np.zeros(32, np.uint8)
    lib().oracle_sha256(_ptr(buf), len(msg), _ptr(out))
    return out.tobytes()


def chunk_digest(tokens: np.ndarray) -> bytes:
    """c = SHA-256(little-endian int32 serialisation of the chunk's tokens)."""
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    out = np.zeros(32, np.uint8)
    lib().oracle_chunk_digest(_ptr(t) if t.size else 0, t.size, _ptr(out))
    return out.tobytes()


def chain_step(prev: bytes, d: bytes, c: bytes) -> bytes:
    """k_i = SHA-256(k_{i-1} || d || c_i)."""
    a = [np.frombuffer(x, np.uint8).copy() for x in (prev, d, c)]
    assert all(x.size == 32 for x in a)
    out = np.zeros(32, np.uint8)
    lib().oracle_chain_step(_ptr(a[0]), _ptr(a[1]), _ptr(a[2]), _ptr(out))
    return out.tobytes()


def request_keys(tokens: np.ndarray, C: int, d: bytes) -> np.ndarray:
    """Keys of one request: uint8[floor(T/C), 32]."""
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    n = t.size // C
    out = np.zeros((max(n, 1), 32), np.uint8)
    dd = np.frombuffer(d, np.uint8).copy()
    got = lib().oracle_request_keys(_ptr(t) if t.size else 0, t.size, C, _ptr(dd), _ptr(out))
    assert got == n
    return out[:n]


def derive_keys(tokens: np.ndarray, tok_off: np.ndarray, C: int, desc_idx: np.ndarray,
                digests: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """All keys of a batch -> (key_off int64[R+1], keys uint8[N, 32])."""
    tokens = np.ascontiguousarray(tokens, dtype=np.int32)
    tok_off = np.ascontiguousarray(tok_off, dtype=np.int64)
    desc_idx = np.ascontiguousarray(desc_idx, dtype=np.uint32)
    digests = np.ascontiguousarray(digests, dtype=np.uint8).reshape(-1, 32)
    R = tok_off.size - 1
    if C <= 0:
        raise OracleError(PK_ERR_ARG, "chunk size must be positive")
    lens = np.diff(tok_off)
    N = int((lens // C).sum()) if R > 0 else 0
    key_off = np.zeros(R + 1, np.int64)
    keys = np.zeros((max(N, 1), 32), np.uint8)
    got = lib().oracle_derive_keys(_ptr(tokens) if tokens.size else 0, _ptr(tok_off), R, C,
                                   _ptr(desc_idx) if R else 0, _ptr(digests) if digests.size else 0,
                                   digests.shape[0], _ptr(key_off), _ptr(keys))
    if got < 0:
        raise OracleError(PK_ERR_ARG, "bad offsets or descriptor index")
    assert got == N
    return key_off, keys[:N]


def request_keys_hashlib(tokens: np.ndarray, C: int, d: bytes) -> np.ndarray:
    """request_keys restated with the standard library's SHA-256 (OpenSSL):
    c_i over the little-endian int32 bytes of chunk i, k_i = H(k_{i-1} || d || c_i)
    from 32 zero bytes.  An independent second implementation of the chain,
    and the CPU baseline that may use the host's SHA-2 instructions."""
    import hashlib
    raw = np.ascontiguousarray(tokens, dtype="<i4").tobytes()
    n = len(raw) // (4 * C)
    out = np.zeros((n, 32), np.uint8)
    prev = bytes(32)
    for i in range(n):
        c = hashlib.sha256(raw[4 * C * i: 4 * C * (i + 1)]).digest()
        prev = hashlib.sha256(prev + bytes(d) + c).digest()
        out[i] = np.frombuffer(prev, np.uint8)
    return out


def derive_keys_hashlib(tokens: np.ndarray, tok_off: np.ndarray, C: int, desc_idx: np.ndarray,
                        digests: np.ndarray, requests=None) -> np.ndarray:
    """Keys of the given requests (default: all), concatenated, by request_keys_hashlib."""
    tok_off = np.asarray(tok_off, np.int64)
    digests = np.asarray(digests, np.uint8).reshape(-1, 32)
    rows = [request_keys_hashlib(tokens[tok_off[r]:tok_off[r + 1]], C, digests[int(desc_idx[r])].tobytes())
            for r in (range(tok_off.size - 1) if requests is None else requests)]
    return np.concatenate(rows) if rows else np.zeros((0, 32), np.uint8)


# --------------------------------------------------------------------------
# Descriptor canonicalisation and enc (Sec. 5.2, 5.3)
# --------------------------------------------------------------------------
def _as_bytes(v) -> bytes:
    if v is None:
        return b""
    if isinstance(v, str):
        return v.encode("utf-8")
    return bytes(v)


def _ascii_lower(b: bytes) -> bytes:
    return bytes(c + 32 if 65 <= c <= 90 else c for c in b)


def canonicalize(desc: Mapping) -> tuple[bytes, ...]:
    """Resolved, injective identities for registry v1 (+ appended extra fields).

    ``desc`` maps the six registry names to str/bytes (absent == empty) and may
    carry ``extra``: a sequence of appended field values (Prop. 1).
    """
    fields = []
    for name in REGISTRY_V1:
        v = _as_bytes(desc.get(name, b""))
        if name in _RESOLVED_FIELDS:
            v = _ascii_lower(v)
            s = v.decode("latin-1")
            v = _SYNONYMS.get(s, s).encode("latin-1")
            if v == b"" or v == b"auto":
                raise OracleError(PK_ERR_UNRESOLVED, f"{name} must be a resolved value")
        if len(v) > MAX_FIELD_BYTES:
            raise OracleError(PK_ERR_FIELD_TOO_LONG, name)
        fields.append(v)
    for v in desc.get("extra", ()) or ():
        v = _as_bytes(v)
        if len(v) > MAX_FIELD_BYTES:
            raise OracleError(PK_ERR_FIELD_TOO_LONG, "extra")
        fields.append(v)
    return tuple(fields)


def enc(fields: Sequence[bytes]) -> bytes:
    """LE32(number of fields) || for each field: LE32(length) || bytes."""
    out = bytearray(len(fields).to_bytes(4, "little"))
    for f in fields:
        f = bytes(f)
        out += len(f).to_bytes(4, "little")
        out += f
    return bytes(out)


def descriptor_digest(desc: Mapping) -> bytes:
    """d = SHA-256(enc(canonicalize(desc)))."""
    return sha256(enc(canonicalize(desc)))


# ---------------------------------------------------------------------------
# Two-level variant.  Sec. 2.2: adapter identity and sharing domain (salt) are
# request-level, weight precision, weight version and KV representation
# worker-level, and the contract binds the two levels through separate
# digests.  Sec. 5.3: the worker-level digest is computed once at startup over
# the resolved values and folded into the model identity; the request-level
# binding is inert for a request carrying neither adapter nor salt, which then
# keys exactly as without it, and the two halves compose independently.  Both
# halves are serialised by the same enc and reduced by the same H.
# ---------------------------------------------------------------------------
WORKER_FIELDS = ("model_id", "weight_precision", "weight_version", "kv_format")
REQUEST_FIELDS = ("adapter_id", "salt")


def worker_half(desc: Mapping) -> tuple[bytes, ...]:
    """The canonical worker-level identities (model id folded in with them;
    the request fields are not read)."""
    worker_only = {n: desc.get(n, b"") for n in WORKER_FIELDS}
    c = dict(zip(REGISTRY_V1, canonicalize(worker_only)))
    return tuple(c[n] for n in WORKER_FIELDS)


def request_half(desc: Mapping) -> tuple[bytes, ...]:
    """The request-level identities: adapter, salt, then appended dimensions
    (opaque bytes; the worker fields are not read)."""
    fields = [_as_bytes(desc.get(n, b"")) for n in REQUEST_FIELDS]
    fields += [_as_bytes(v) for v in (desc.get("extra", ()) or ())]
    for v in fields:
        if len(v) > MAX_FIELD_BYTES:
            raise OracleError(PK_ERR_FIELD_TOO_LONG, "request field")
    return tuple(fields)


def worker_digest(desc: Mapping) -> bytes:
    """d_w = H(enc(worker half))."""
    return sha256(enc(worker_half(desc)))


def request_digest(d_w: bytes, desc: Mapping) -> bytes:
    """The digest a request's keys fold in: d_w itself when the request half
    is empty (the binding is inert), else H(d_w || H(enc(request half)))."""
    q = request_half(desc)
    if all(len(f) == 0 for f in q) and len(q) == len(REQUEST_FIELDS):
        return bytes(d_w)
    return sha256(bytes(d_w) + sha256(enc(q)))


def two_level_digests(descs: Iterable[Mapping]) -> np.ndarray:
    """uint8[D][32]: request_digest(worker_digest(d), d) for each descriptor."""
    descs = list(descs)
    out = np.zeros((len(descs), 32), np.uint8)
    for j, d in enumerate(descs):
        out[j] = np.frombuffer(request_digest(worker_digest(d), d), np.uint8)
    return out


def descriptor_digests(descs: Iterable[Mapping]) -> np.ndarray:
    ds = [descriptor_digest(d) for d in descs]
    if not ds:
        return np.zeros((0, 32), np.uint8)
    return np.frombuffer(b"".join(ds), np.uint8).reshape(-1, 32).copy()


# --------------------------------------------------------------------------
# Table semantics
# --------------------------------------------------------------------------
def prefix128(keys: np.ndarray) -> np.ndarray:
    """First 16 bytes of each key (standard digest byte order)."""
    keys = np.ascontiguousarray(keys, dtype=np.uint8)
    return np.ascontiguousarray(keys.reshape(-1, keys.shape[-1])[:, :16])


class DictTable:
    """Exact-match map from 16-byte key prefixes to uint32 slots.

    Capacity rule: at most ``capacity - 1`` entries (one slot always stays
    empty); an insertion that would exceed it is refused with TABLE_FULL.
    The all-zero prefix is the empty marker and cannot be stored.
    """

    def __init__(self, capacity: int):
        if capacity < 2 or capacity & (capacity - 1):
            raise OracleError(PK_ERR_CAPACITY, "capacity must be a power of two >= 2")
        self.capacity = capacity
        self.map: dict[bytes, int] = {}

    def __len__(self):
        return len(self.map)

    def store(self, keys: np.ndarray, slots: np.ndarray):
        """Insert in array order -> (result int32[n], slot_out uint32[n])."""
        p = prefix128(keys)
        slots = np.asarray(slots, dtype=np.uint32)
        n = p.shape[0]
        result = np.zeros(n, np.int32)
        slot_out = np.full(n, NO_SLOT, np.uint32)
        zero = bytes(16)
        for i in range(n):
            k = p[i].tobytes()
            if k == zero:
                result[i] = PK_ERR_RESERVED_KEY
                continue
            if int(slots[i]) == NO_SLOT:
                result[i] = PK_ERR_ARG
                continue
            if k in self.map:
                result[i] = STORE_PRESENT
                slot_out[i] = self.map[k]
            elif len(self.map) + 1 >= self.capacity:
                result[i] = PK_ERR_TABLE_FULL
            else:
                self.map[k] = int(slots[i])
                result[i] = STORE_INSERTED
                slot_out[i] = int(slots[i])
        return result, slot_out

    def get(self, keys: np.ndarray) -> np.ndarray:
        p = prefix128(keys)
        return np.array([self.map.get(p[i].tobytes(), NO_SLOT) for i in range(p.shape[0])],
                        dtype=np.uint32)


class SortedTable:
    """Same semantics as DictTable, computed with sort / searchsorted.

    Holds unique prefixes sorted bytewise with the slot of each one's first
    insertion.  Used for tables of millions of entries.
    """

    def __init__(self, capacity: int):
        if capacity < 2 or capacity & (capacity - 1):
            raise OracleError(PK_ERR_CAPACITY, "capacity must be a power of two >= 2")
        self.capacity = capacity
        self.keys = np.zeros(0, dtype="V16")
        self.slots = np.zeros(0, np.uint32)

    def __len__(self):
        return int(self.keys.size)

    @staticmethod
    def _v16(keys: np.ndarray) -> np.ndarray:
        return prefix128(keys).view("V16").reshape(-1)

    def _find(self, q: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
        if self.keys.size == 0:
            return np.zeros(q.size, bool), np.zeros(q.size, np.int64)
        pos = np.searchsorted(self.keys, q)
        posc = np.minimum(pos, self.keys.size - 1)
        found = self.keys[posc] == q
        return found, posc

    def get(self, keys: np.ndarray) -> np.ndarray:
        q = self._v16(keys)
        found, pos = self._find(q)
        out = np.full(q.size, NO_SLOT, np.uint32)
        out[found] = self.slots[pos[found]]
        return out

    def store(self, keys: np.ndarray, slots: np.ndarray):
        q = self._v16(keys)
        slots = np.asarray(slots, dtype=np.uint32)
        n = q.size
        result = np.zeros(n, np.int32)
        slot_out = np.full(n, NO_SLOT, np.uint32)
        zero = np.zeros(1, dtype="V16")[0]
        bad_key = q == zero
        bad_slot = slots == NO_SLOT
        result[bad_key] = PK_ERR_RESERVED_KEY
        result[bad_slot & ~bad_key] = PK_ERR_ARG
        ok = ~(bad_key | bad_slot)
        found, pos = self._find(q)
        pre = ok & found
        result[pre] = STORE_PRESENT
        slot_out[pre] = self.slots[pos[pre]]
        new = np.nonzero(ok & ~found)[0]
        if new.size:
            uq, first, inv = np.unique(q[new], return_index=True, return_inverse=True)
            # insertion order of the new distinct keys = order of first occurrence
            order = np.argsort(first, kind="stable")
            room = max(self.capacity - 1 - len(self), 0)
            accepted_rank = np.zeros(uq.size, bool)
            accepted_rank[order[:room]] = True
            win_idx = new[first]                       # batch index of each distinct key's first occurrence
            acc = accepted_rank[inv]
            idx_acc = new[acc]
            is_first = idx_acc == win_idx[inv[acc]]
            result[idx_acc[is_first]] = STORE_INSERTED
            result[idx_acc[~is_first]] = STORE_PRESENT
            slot_out[idx_acc] = slots[win_idx[inv[acc]]]
            result[new[~acc]] = PK_ERR_TABLE_FULL
            ins_keys = uq[accepted_rank]
            ins_slots = slots[win_idx[accepted_rank]]
            allk = np.concatenate([self.keys, ins_keys])
            alls = np.concatenate([self.slots, ins_slots])
            o = np.argsort(allk, kind="stable")
            self.keys, self.slots = allk[o], alls[o]
        return result, slot_out


def lookup(table, keys: np.ndarray, key_off: np.ndarray):
    """Probe every key -> (hit_chunks int32[R], slots uint32[N]).

    hit_chunks[r] = h_r, the largest j such that chunks 0..j-1 of request r are
    all present; slots[i] is the stored slot of key i or NO_SLOT.
    """
    key_off = np.asarray(key_off, dtype=np.int64)
    R = key_off.size - 1
    slots = table.get(keys) if keys.shape[0] else np.zeros(0, np.uint32)
    hit = np.zeros(R, np.int32)
    for r in range(R):
        s = slots[key_off[r]:key_off[r + 1]]
        miss = np.nonzero(s == NO_SLOT)[0]
        hit[r] = int(miss[0]) if miss.size else s.size
    return hit, slots


def store_misses(table, keys: np.ndarray, key_off: np.ndarray, hit_chunks: np.ndarray,
                 slots: np.ndarray):
    """Store the keys of every miss range [h_r, n_r), in global key order.

    Returns (result int32[N], slot_out uint32[N]); entries below h_r are SKIPPED.
    """
    key_off = np.asarray(key_off, dtype=np.int64)
    N = keys.shape[0]
    idx = []
    for r in range(key_off.size - 1):
        idx.extend(range(int(key_off[r]) + int(hit_chunks[r]), int(key_off[r + 1])))
    idx = np.asarray(idx, dtype=np.int64)
    result = np.full(N, STORE_SKIPPED, np.int32)
    slot_out = np.full(N, NO_SLOT, np.uint32)
    if idx.size:
        res, so = table.store(keys[idx], np.asarray(slots, np.uint32)[idx])
        result[idx] = res
        slot_out[idx] = so
    return result, slot_out


def seed_table(table, seed_keys: np.ndarray, filler: np.ndarray, target_entries: int):
    """Pre-fill a table: the seed keys in order (slot = list index), then filler
    keys, continuing the index, until it holds ``target_entries`` entries."""
    n_seed = seed_keys.shape[0]
    if n_seed:
        table.store(seed_keys, np.arange(n_seed, dtype=np.uint32))
    need = target_entries - len(table)
    if need > 0:
        if need > filler.shape[0]:
            raise OracleError(PK_ERR_ARG, "not enough filler keys")
        table.store(filler[:need], np.arange(n_seed, n_seed + need, dtype=np.uint32))
    return table


# ---------------------------------------------------------------------------
# Store-side differential omission test (Sec. 6.3, omission detection; Eq. 4):
# a key of one worker that a reference worker also wrote, with differing page
# bytes, means the binding omits a dimension that changes the cached state.
# ---------------------------------------------------------------------------
PAGE_ABSENT, PAGE_EQUAL, PAGE_DIFFERS = 0, 1, 2


def compare_pages(slots: np.ndarray, pages: np.ndarray, ref_pages: np.ndarray):
    """Per key j: PAGE_ABSENT if slots[j] is NO_SLOT, else PAGE_EQUAL or
    PAGE_DIFFERS for pages[j] against ref_pages[slots[j]].  Returns
    (verdict int32[n], counts int64[3])."""
    slots = np.asarray(slots, np.uint32)
    verdict = np.zeros(slots.size, np.int32)
    for j, s in enumerate(slots):
        if int(s) != NO_SLOT:
            verdict[j] = PAGE_EQUAL if np.array_equal(pages[j], ref_pages[int(s)]) else PAGE_DIFFERS
    return verdict, np.bincount(verdict, minlength=3).astype(np.int64)


def omission_check(ref_keys: np.ndarray, ref_pages: np.ndarray, keys: np.ndarray, pages: np.ndarray):
    """Join keys to the reference worker's on the 128-bit prefix (the first
    reference page of a repeated key), then compare_pages."""
    cap = 2
    while cap <= ref_keys.shape[0]:
        cap *= 2
    t = DictTable(cap)
    t.store(ref_keys, np.arange(ref_keys.shape[0], dtype=np.uint32))
    return compare_pages(t.get(keys), pages, ref_pages)


# ---------------------------------------------------------------------------
# Content identity (Sec. 5.3: an adapter is bound by an identity of its
# contents, every tensor's name, dtype, shape and bytes with the meaningful
# configuration fields; Sec. 5.1: the identity function is open as long as it
# is injective and stable).  A fixed-shape tree of SHA-256: each level hashes
# every 1 KiB block of the level below, the last block zero-padded (an empty
# buffer is one zero block), until one digest remains.
# ---------------------------------------------------------------------------
TREE_BLOCK = 1024


def tree_level(data: bytes) -> bytes:
    """The digests of the 1 KiB blocks of data (zero-padded), concatenated."""
    m = max(1, -(-len(data) // TREE_BLOCK))
    padded = bytes(data) + bytes(m * TREE_BLOCK - len(data))
    return b"".join(sha256(padded[i * TREE_BLOCK:(i + 1) * TREE_BLOCK]) for i in range(m))


def content_digest(data: bytes) -> bytes:
    """The tree top of data: levels until one 32-byte digest."""
    level = tree_level(bytes(data))
    while len(level) > 32:
        level = tree_level(level)
    return level


def tensor_identity(name, dtype, shape, n_bytes: int, top: bytes) -> bytes:
    """H(enc(name, dtype, shape as LE64 each, LE64(n_bytes), top))."""
    dims = b"".join(int(x).to_bytes(8, "little", signed=True) for x in shape)
    return sha256(enc([_as_bytes(name), _as_bytes(dtype), dims, int(n_bytes).to_bytes(8, "little"), bytes(top)]))


def adapter_identity(tensor_ids, config) -> bytes:
    """H(enc(enc(config fields), tensor identities in the given order))."""
    return sha256(enc([enc([_as_bytes(c) for c in config])] + [bytes(t) for t in tensor_ids]))


# ---------------------------------------------------------------------------
# Connector key strings (Sec. 5.3, connector integration): a fixed-width text
# key carries the 128-bit digest as twenty-two base64 characters and the model
# identity with the worker provenance as a fixed-length hash.  Readings: the
# alphabet is the standard one of RFC 4648, Sec. 4, without the "=" padding;
# the fixed-length hash is the first 16 bytes of the worker digest d_w, in
# the same 22-character form; a key string row is prefix || 22 characters ||
# zero bytes up to the row width.
# ---------------------------------------------------------------------------
B64_ALPHABET = "ABCDEFGHIJKLMNOPQRSTUVWXYZabcdefghijklmnopqrstuvwxyz0123456789+/"
KEY_STRING_CHARS = 22


def base64_encode(data: bytes) -> str:
    """RFC 4648, Sec. 4: each 24-bit group of input bits (most significant
    first) is four 6-bit indices into the alphabet; a final group of 8 or 16
    bits is zero-extended to 12 or 18 bits and followed by "==" or "="."""
    data = bytes(data)
    out = []
    for i in range(0, len(data), 3):
        group = data[i:i + 3]
        bits = int.from_bytes(group, "big") << (8 * (3 - len(group)))
        chars = [B64_ALPHABET[(bits >> (18 - 6 * j)) & 63] for j in range(4)]
        n_chars = len(group) + 1  # 1 byte -> 2 characters, 2 -> 3, 3 -> 4
        out.append("".join(chars[:n_chars]) + "=" * (4 - n_chars))
    return "".join(out)


def key_string(prefix16: bytes) -> str:
    """The 22-character form of a 128-bit key prefix: base64 without "=="."""
    prefix16 = bytes(prefix16)
    if len(prefix16) != 16:
        raise OracleError(PK_ERR_ARG, "a key prefix is 16 bytes")
    s = base64_encode(prefix16)
    assert s.endswith("==")
    return s[:KEY_STRING_CHARS]


def model_tag(desc: Mapping) -> str:
    """The fixed-length hash over the model identity and worker provenance."""
    return key_string(worker_digest(desc)[:16])


def key_strings(keys: np.ndarray, prefix: bytes, width: int) -> np.ndarray:
    """uint8[n, width]: row i = prefix || key_string(keys[i, :16]) || zeros."""
    prefix = bytes(prefix)
    if len(prefix) + KEY_STRING_CHARS > width:
        raise OracleError(PK_ERR_ARG, "row narrower than prefix + 22 characters")
    keys = np.asarray(keys, np.uint8).reshape(-1, 32)
    out = np.zeros((keys.shape[0], width), np.uint8)
    for i in range(keys.shape[0]):
        row = prefix + key_string(keys[i, :16].tobytes()).encode("ascii")
        out[i, :len(row)] = np.frombuffer(row, np.uint8)
    return out


# ---------------------------------------------------------------------------
# Eviction under a fixed budget (Sec. 6.5: binding provenance keeps one copy
# per provenance, so a store of fixed size evicts more and thrashes once the
# distinct working set exceeds it).  Readings: the budget counts entries
# (chunks); recency is least-recently-used with a last-use stamp
# (n << 32) | e per entry, n the store call's number on the table and e the
# key's index in the call; a call uses every key that was in the table at its
# start or that it stores with a valid slot; eviction runs between calls and,
# when the table holds more than `budget` entries, removes every entry whose
# stamp is at most the (keep+1)-th largest (the least recently used, down to
# `keep`; a group of equal stamps, possible only for never-used entries at
# stamp 0, goes as a whole).
# ---------------------------------------------------------------------------
class BudgetTable:
    """DictTable plus last-use stamps and the store-call counter."""

    def __init__(self, capacity: int):
        self.table = DictTable(capacity)
        self.stamps: dict[bytes, int] = {}
        self.calls = 0

    def __len__(self):
        return len(self.table)

    def _use(self, k: bytes, e: int) -> None:
        s = (self.calls << 32) | e
        if s > self.stamps.get(k, 0):
            self.stamps[k] = s

    def store(self, keys: np.ndarray, slots: np.ndarray):
        """List-mode store; every entry that ends INSERTED or PRESENT is a use."""
        self.calls += 1
        res, so = self.table.store(keys, slots)
        p = prefix128(keys)
        for e in range(p.shape[0]):
            if res[e] in (STORE_INSERTED, STORE_PRESENT):
                self._use(p[e].tobytes(), e)
        return res, so

    def lookup_store(self, keys: np.ndarray, key_off: np.ndarray, new_slots: np.ndarray):
        """Lookup, then the store of every miss range (one call)."""
        self.calls += 1
        p = prefix128(keys)
        new_slots = np.asarray(new_slots, np.uint32)
        present0 = self.table.get(keys) != NO_SLOT if p.shape[0] else np.zeros(0, bool)
        hit, slots = lookup(self.table, keys, key_off)
        res, so = store_misses(self.table, keys, key_off, hit, new_slots)
        for e in range(p.shape[0]):
            k = p[e].tobytes()
            if present0[e] or (int(new_slots[e]) != NO_SLOT and k in self.table.map):
                self._use(k, e)
        return hit, slots, res, so

    def evict(self, budget: int, keep: int) -> np.ndarray:
        """Sorted uint32 slots of the removed entries (empty within the budget)."""
        if keep > budget:
            raise OracleError(PK_ERR_ARG, "keep > budget")
        m = self.table.map
        if len(m) <= budget or len(m) <= keep:
            return np.zeros(0, np.uint32)
        v = sorted((self.stamps.get(k, 0) for k in m), reverse=True)[keep]
        gone = [k for k in m if self.stamps.get(k, 0) <= v]
        out = np.array(sorted(m[k] for k in gone), np.uint32)
        for k in gone:
            del m[k]
            self.stamps.pop(k, None)
        return out

    def triples(self):
        """Sorted (16-byte key, slot, stamp) of every entry."""
        return sorted((k, s, self.stamps.get(k, 0)) for k, s in self.table.map.items())
