"""Seeded synthetic workloads shaped like the paper's serving setups.

This module holds no part of the key derivation: it only draws token ids,
request offsets, descriptor field values and random filler keys.  Both the
CUDA path and the CPU oracle consume its output.

The paper's public workloads (ShareGPT prompts paired with system prompts,
Sec. 4.1) are not available; these configurations stand in with the shapes the
paper describes: shared system / document prefixes, multi-adapter serving,
mixed weight precision, several KV formats and weight versions, and several
sharing-domain salts (Sec. 2.2, Sec. 4.5).

Every array comes from ``numpy.random.default_rng(seed)`` (PCG64) in a fixed
draw order, so a configuration is reproducible from its seed alone.  Filler
table keys come from ``default_rng(seed + 1000)`` and are distinct and
non-zero.

A table is pre-filled ("seeded") from a *prior* batch: the keys of its
requests (optionally only the first ``prior_chunks`` chunks of each), in
global key order with slot = position in that list, followed by filler keys
(continuing the position count) until the table holds ``target_entries``
entries.  Each side computes the prior batch's keys itself.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional
import zlib

import numpy as np

REGISTRY_V1 = ("model_id", "weight_precision", "weight_version", "adapter_id", "kv_format", "salt")
MODEL_ID = "synthetic/model-7b"
KV_FORMATS = ("bf16", "fp16", "fp8_e4m3", "fp8_e5m2")
PRECISIONS = ("bf16", "fp8_e4m3")


@dataclass
class Batch:
    tokens: np.ndarray      # int32[total tokens]
    tok_off: np.ndarray     # int64[R + 1]; request r is tokens[tok_off[r]:tok_off[r+1]]
    desc_idx: np.ndarray    # uint32[R]; index into Workload.descriptors

    @property
    def R(self) -> int:
        return int(self.tok_off.size - 1)

    @property
    def n_tokens(self) -> int:
        return int(self.tokens.size)

    def n_chunks(self, C: int) -> np.ndarray:
        return np.diff(self.tok_off) // C

    def select(self, rows) -> "Batch":
        rows = np.asarray(rows, dtype=np.int64)
        parts = [self.tokens[self.tok_off[r]:self.tok_off[r + 1]] for r in rows]
        lens = np.array([p.size for p in parts], dtype=np.int64)
        off = np.zeros(rows.size + 1, np.int64)
        np.cumsum(lens, out=off[1:])
        toks = np.concatenate(parts).astype(np.int32) if parts else np.zeros(0, np.int32)
        return Batch(toks, off, self.desc_idx[rows].astype(np.uint32))


@dataclass
class Workload:
    name: str
    chunk_tokens: int
    descriptors: list            # list of dict(field name -> str)
    batch: Batch
    prior: Optional[Batch]       # batch whose keys seed the table
    prior_chunks: Optional[int]  # keep only the first k chunks per prior request (None: all)
    filler: np.ndarray           # uint8[F, 16]
    capacity_log2: int
    target_entries: int
    expected_hits: Optional[np.ndarray] = None   # h_r where the construction fixes it
    notes: dict = field(default_factory=dict)

    @property
    def capacity(self) -> int:
        return 1 << self.capacity_log2

    def tokens_keyed(self) -> int:
        return int(self.batch.n_chunks(self.chunk_tokens).sum()) * self.chunk_tokens

    def n_keys(self) -> int:
        return int(self.batch.n_chunks(self.chunk_tokens).sum())


# --------------------------------------------------------------------------
# helpers
# --------------------------------------------------------------------------
def _hex(rng: np.random.Generator, nbytes: int) -> str:
    return bytes(rng.integers(0, 256, nbytes, dtype=np.uint8)).hex()


def _desc(precision="bf16", version="", adapter="", kv="bf16", salt="") -> dict:
    return {"model_id": MODEL_ID, "weight_precision": precision, "weight_version": version,
            "adapter_id": adapter, "kv_format": kv, "salt": salt}


def filler_keys(seed: int, count: int) -> np.ndarray:
    """``count`` distinct, non-zero random 128-bit keys from default_rng(seed)."""
    rng = np.random.default_rng(seed)
    out = rng.integers(0, 256, (count, 16), dtype=np.uint8)
    for _ in range(8):
        v = out.view("V16").reshape(-1)
        _, first = np.unique(v, return_index=True)
        keep = np.zeros(count, bool)
        keep[first] = True
        keep &= out.any(axis=1)
        if keep.all():
            return out
        bad = np.nonzero(~keep)[0]
        out[bad] = rng.integers(0, 256, (bad.size, 16), dtype=np.uint8)
    raise RuntimeError("could not draw distinct filler keys")


def _lengths(rng, R, T, C, ragged) -> np.ndarray:
    if not ragged:
        return np.full(R, T, np.int64)
    # ragged: trailing partial chunks, a few requests shorter than one chunk,
    # a few exact multiples of the chunk size
    lens = T - rng.integers(0, C, R)
    lens[:: max(R // 7, 1)] = T
    if R >= 5:
        lens[3] = rng.integers(0, C)          # no full chunk
    return np.maximum(lens, 0).astype(np.int64)


def _pack(rows) -> tuple[np.ndarray, np.ndarray]:
    lens = np.array([r.size for r in rows], dtype=np.int64)
    off = np.zeros(len(rows) + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    toks = np.concatenate(rows).astype(np.int32) if rows else np.zeros(0, np.int32)
    return toks, off


# --------------------------------------------------------------------------
# configurations
# --------------------------------------------------------------------------
def tiny(seed: int = 0) -> Workload:
    """8 requests x 512 tokens in [0, 32000), chunk 256; 2 adapters x 2 salts;
    64-slot table holding the keys of requests 0-3 plus 8 filler (load 0.25).
    Request 4 repeats request 0's tokens under another adapter (h = 0);
    request 5 repeats request 1 with the same descriptor (h = 2)."""
    rng = np.random.default_rng(seed)
    R, T, C, V = 8, 512, 256, 32000
    toks = rng.integers(0, V, (R, T), dtype=np.int64).astype(np.int32)
    toks[4] = toks[0]
    toks[5] = toks[1]
    version = _hex(rng, 20)
    salts = [_hex(rng, 16), _hex(rng, 16)]
    adapters = ["adapter-00", "adapter-01"]
    descs = [_desc(version=version, adapter=adapters[a], salt=salts[s]) for s in (0, 1) for a in (0, 1)]
    a = np.arange(R) % 2
    s = (np.arange(R) // 2) % 2
    a[4] = 1 - a[0]
    s[4] = s[0]
    desc_idx = (a + 2 * s).astype(np.uint32)
    tokens, off = _pack(list(toks))
    batch = Batch(tokens, off, desc_idx)
    return Workload("tiny", C, descs, batch, batch.select(range(4)), None,
                    filler_keys(seed + 1000, 16), 6, 16,
                    expected_hits=np.array([2, 2, 2, 2, 0, 2, 0, 0], np.int32))


def multi_adapter(seed: int = 1, R: int = 1024, T: int = 4096, capacity_log2: int = 20,
                  load: float = 0.5, ragged: bool = False) -> Workload:
    """Multi-adapter serving: R x T tokens, vocab 152064, chunk 256; requests
    with r % 5 < 2 start with one 2048-token system prefix; descriptors uniform
    over 8 adapters x 2 weight precisions x 2 salts; table at the given load,
    seeded from a prior batch (seed + 100) drawn the same way."""
    rng = np.random.default_rng(seed)
    C, V, S_len = 256, 152064, 2048
    version = _hex(rng, 20)
    salts = [_hex(rng, 16), _hex(rng, 16)]
    descs = [_desc(precision=PRECISIONS[p], version=version, adapter=f"adapter-{a:02d}", salt=salts[s])
             for a in range(8) for p in range(2) for s in range(2)]
    S = rng.integers(0, V, S_len, dtype=np.int64).astype(np.int32)

    def draw(r_rng):
        lens = _lengths(r_rng, R, T, C, ragged)
        rows = []
        for r in range(R):
            row = r_rng.integers(0, V, int(lens[r]), dtype=np.int64).astype(np.int32)
            if r % 5 < 2 and row.size >= S_len:
                row[:S_len] = S
            rows.append(row)
        desc_idx = r_rng.integers(0, len(descs), R).astype(np.uint32)
        toks, off = _pack(rows)
        return Batch(toks, off, desc_idx)

    batch = draw(rng)
    prior = draw(np.random.default_rng(seed + 100))
    cap = 1 << capacity_log2
    target = int(load * cap)
    return Workload("multi_adapter", C, descs, batch, prior, None,
                    filler_keys(seed + 1000, target), capacity_log2, target)


def small_block(seed: int = 2, R: int = 16384, T: int = 2048, capacity_log2: int = 23,
                load: float = 0.6, n_templates: int = 256, ragged: bool = False) -> Workload:
    """Small-block paged cache: R x T tokens, chunk 16, vocab 128256.  Each
    request copies a prefix [0, L_t) of one of 256 templates (template rank k
    drawn with probability proportional to k^-1.1, L_t uniform in 16..T) and is
    random afterwards.  Descriptors uniform over 4 KV formats x 4 weight
    versions.  Table seeded from a prior batch (seed + 100)."""
    rng = np.random.default_rng(seed)
    C, V = 16, 128256
    versions = [_hex(rng, 20) for _ in range(4)]
    descs = [_desc(version=versions[v], kv=KV_FORMATS[k]) for k in range(4) for v in range(4)]
    templates = rng.integers(0, V, (n_templates, T), dtype=np.int64).astype(np.int32)
    shared = rng.integers(16, T + 1, n_templates)
    w = np.arange(1, n_templates + 1, dtype=np.float64) ** -1.1
    w /= w.sum()

    def draw(r_rng):
        lens = _lengths(r_rng, R, T, C, ragged)
        t = r_rng.choice(n_templates, size=R, p=w)
        rnd = r_rng.integers(0, V, (R, T), dtype=np.int64).astype(np.int32)
        mask = np.arange(T)[None, :] < shared[t][:, None]
        full = np.where(mask, templates[t], rnd)
        rows = [full[r, :lens[r]] for r in range(R)]
        desc_idx = r_rng.integers(0, len(descs), R).astype(np.uint32)
        toks, off = _pack(rows)
        return Batch(toks, off, desc_idx)

    batch = draw(rng)
    prior = draw(np.random.default_rng(seed + 100))
    cap = 1 << capacity_log2
    target = int(load * cap)
    return Workload("small_block", C, descs, batch, prior, None,
                    filler_keys(seed + 1000, target), capacity_log2, target)


def long_context(seed: int = 3, R: int = 64, T: int = 131072, n_shared: int = 16,
                 shared_len: int = 65536, capacity_log2: int = 22, load: float = 0.5,
                 ragged: bool = False) -> Workload:
    """Long context: R x T tokens, chunk 256, vocab 152064; requests 0..15 share
    a 65536-token document prefix; one adapter, salt = r % 4.  The table holds
    the keys of each request's first half of chunks plus filler, so about half
    of all probes hit (every request's h_r is half its chunk count)."""
    rng = np.random.default_rng(seed)
    C, V = 256, 152064
    version = _hex(rng, 20)
    salts = [_hex(rng, 16) for _ in range(4)]
    descs = [_desc(version=version, adapter="adapter-00", salt=salts[s]) for s in range(4)]
    doc = rng.integers(0, V, shared_len, dtype=np.int64).astype(np.int32)
    lens = _lengths(rng, R, T, C, ragged)
    rows = []
    for r in range(R):
        row = rng.integers(0, V, int(lens[r]), dtype=np.int64).astype(np.int32)
        if r < n_shared and row.size >= shared_len:
            row[:shared_len] = doc
        rows.append(row)
    desc_idx = (np.arange(R) % 4).astype(np.uint32)
    toks, off = _pack(rows)
    batch = Batch(toks, off, desc_idx)
    half = (T // C) // 2
    cap = 1 << capacity_log2
    target = int(load * cap)
    expected = None if ragged else np.full(R, half, np.int32)
    return Workload("long_context", C, descs, batch, batch, half,
                    filler_keys(seed + 1000, target), capacity_log2, target,
                    expected_hits=expected)


def provenance_sweep(D: int, seed: int = 4, R: int = 4096, T: int = 8192, prefix_len: int = 4096,
                     capacity_log2: int = 24, load: float = 0.7, ragged: bool = False) -> Workload:
    """Provenance-diversity sweep: R x T tokens, chunk 256; one token-identical
    4096-token prefix P; request r uses descriptor r % D, the D descriptors
    differing in adapter / weight precision / weight version / KV format / salt.
    The table holds P's 16 chunk keys under each of the D descriptors plus
    filler, so every request hits its first 16 chunks and misses the rest
    (half the lookups negative)."""
    rng = np.random.default_rng(seed)
    C, V = 256, 152064
    versions = [_hex(rng, 20) for _ in range(4)]
    salts = [""] + [_hex(rng, 16) for _ in range(3)]
    adapters = [""] + [f"adapter-{a:02d}" for a in range(8)]
    combos = [(a, p, v, k, s) for a in range(9) for p in range(2) for v in range(4)
              for k in range(4) for s in range(4)]
    pick = rng.choice(len(combos), size=D, replace=False)
    descs = []
    for j in pick:
        a, p, v, k, s = combos[int(j)]
        descs.append(_desc(precision=PRECISIONS[p], version=versions[v], adapter=adapters[a],
                           kv=KV_FORMATS[k], salt=salts[s]))
    P = rng.integers(0, V, prefix_len, dtype=np.int64).astype(np.int32)
    lens = _lengths(rng, R, T, C, ragged)
    rows = []
    for r in range(R):
        row = rng.integers(0, V, int(lens[r]), dtype=np.int64).astype(np.int32)
        if row.size >= prefix_len:
            row[:prefix_len] = P
        rows.append(row)
    desc_idx = (np.arange(R) % D).astype(np.uint32)
    toks, off = _pack(rows)
    batch = Batch(toks, off, desc_idx)
    ptoks, poff = _pack([P.copy() for _ in range(D)])
    prior = Batch(ptoks, poff, np.arange(D, dtype=np.uint32))
    cap = 1 << capacity_log2
    target = int(load * cap)
    expected = None if ragged else np.full(R, prefix_len // C, np.int32)
    return Workload(f"provenance_sweep_D{D}", C, descs, batch, prior, None,
                    filler_keys(seed + 1000, target), capacity_log2, target,
                    expected_hits=expected, notes={"D": D})


FULL_CONFIGS = {
    "tiny": tiny,
    "multi_adapter": multi_adapter,
    "small_block": small_block,
    "long_context": long_context,
    "provenance_sweep_D1": lambda: provenance_sweep(1),
    "provenance_sweep_D4": lambda: provenance_sweep(4),
    "provenance_sweep_D16": lambda: provenance_sweep(16),
    "provenance_sweep_D64": lambda: provenance_sweep(64),
}


def reduced(name: str) -> Workload:
    """Scaled-down, ragged variants that the oracle finishes in seconds while
    still spanning many thread blocks and partial trailing chunks."""
    if name == "tiny":
        return tiny()
    if name == "multi_adapter":
        return multi_adapter(R=40, T=4096, capacity_log2=12, ragged=True)
    if name == "small_block":
        return small_block(R=300, T=512, capacity_log2=14, n_templates=32, ragged=True)
    if name == "long_context":
        return long_context(R=6, T=8192, n_shared=3, shared_len=4096, capacity_log2=10,
                            ragged=True)
    if name.startswith("provenance_sweep_D"):
        D = int(name[len("provenance_sweep_D"):])
        return provenance_sweep(D, R=max(2 * D, 24), T=2048, prefix_len=1024,
                                capacity_log2=12, ragged=True)
    raise KeyError(name)


def seed_list(prior_keys: np.ndarray, prior_key_off: np.ndarray, prior_chunks: Optional[int]) -> np.ndarray:
    """Select the seed keys of a prior batch: all, or the first ``prior_chunks``
    of each request, in global key order.  Pure indexing."""
    if prior_chunks is None:
        return prior_keys
    idx = []
    for r in range(prior_key_off.size - 1):
        a, b = int(prior_key_off[r]), int(prior_key_off[r + 1])
        idx.append(np.arange(a, min(b, a + prior_chunks)))
    idx = np.concatenate(idx) if idx else np.zeros(0, np.int64)
    return prior_keys[idx]


# ---------------------------------------------------------------------------
# Synthetic KV pages for the store-side omission test (sec. 6.3: two workers
# that differ in one dimension write the same documents into one store).  No
# model runs here: the bytes of the page of chunk i of a request are a
# deterministic pseudo-random function of the request's tokens up to the end of
# chunk i (its prefix, which the state of that chunk depends on) and of the
# computational dimensions of the worker that wrote it (model id, weight
# precision, weight version, adapter, KV format).  The salt changes who may
# reuse state, not the state (sec. 2.2), so it does not enter the bytes.  The
# seeding uses CRC-32, not the keys' hash.
# ---------------------------------------------------------------------------
COMPUTATIONAL_FIELDS = ("model_id", "weight_precision", "weight_version", "adapter_id", "kv_format")


def _config_seed(desc: dict) -> int:
    blob = "\x1f".join(str(desc.get(f, "")) for f in COMPUTATIONAL_FIELDS).encode()
    return zlib.crc32(blob)


def kv_pages(batch: Batch, C: int, desc_of_request, page_bytes: int) -> np.ndarray:
    """uint8[N_chunks, page_bytes], in key order (request by request, chunk by
    chunk): the page each full chunk would write.  desc_of_request(r) gives the
    descriptor of the worker configuration that served request r."""
    assert page_bytes % 16 == 0
    pages = []
    for r in range(batch.R):
        row = batch.tokens[batch.tok_off[r]:batch.tok_off[r + 1]]
        cfg = _config_seed(desc_of_request(r))
        crc = 0
        for i in range(row.size // C):
            crc = zlib.crc32(row[i * C:(i + 1) * C].astype("<i4").tobytes(), crc)
            rng = np.random.default_rng([crc, cfg])
            pages.append(rng.integers(0, 256, page_bytes, dtype=np.uint8))
    return np.stack(pages) if pages else np.zeros((0, page_bytes), np.uint8)


@dataclass
class OmissionCase:
    """Worker A and worker B (A with one dimension changed) serving the same
    documents; keys are bound with `binding` (the descriptor fields the key
    covers), pages follow each worker's full configuration."""
    name: str
    chunk_tokens: int
    batch: Batch
    worker_a: dict
    worker_b: dict
    bound_a: dict
    bound_b: dict
    pages_a: np.ndarray
    pages_b: np.ndarray


def omission_case(varied: str, omit: Optional[str], seed: int = 5, R: int = 12, T: int = 640, C: int = 64,
                  page_bytes: int = 256) -> OmissionCase:
    """`varied`: the dimension in which worker B differs from A; `omit`: the
    dimension the key binding leaves out (None: the complete binding).  Omitting
    a field means both workers' key descriptors carry the same fixed value for
    it."""
    rng = np.random.default_rng(seed)
    a = _desc(precision="bf16", version=_hex(rng, 20), adapter="adapter-00", kv="bf16", salt="tenant-a")
    changed = {"model_id": MODEL_ID + "-v2", "weight_precision": "fp8_e4m3", "weight_version": _hex(rng, 20),
               "adapter_id": "adapter-01", "kv_format": "fp8_e5m2", "salt": "tenant-b"}
    b = dict(a, **{varied: changed[varied]})
    lens = _lengths(rng, R, T, C, True)
    rows = [rng.integers(0, 32000, int(n), dtype=np.int64).astype(np.int32) for n in lens]
    toks, off = _pack(rows)
    batch = Batch(toks, off, np.zeros(R, np.uint32))

    def bound(d):
        if omit is None:
            return dict(d)
        fixed = {"weight_precision": "bf16", "kv_format": "bf16"}.get(omit, "")
        return dict(d, **{omit: fixed})
    return OmissionCase(f"vary {varied}, omit {omit}", C, batch, a, b, bound(a), bound(b),
                        kv_pages(batch, C, lambda r: a, page_bytes), kv_pages(batch, C, lambda r: b, page_bytes))


# --------------------------------------------------------------------------
# Eviction under a fixed budget (Sec. 6.5): one pool of prompts served under
# D provenances (adapters) in turn, against a store whose budget holds about
# one copy of the pool's chunks.  Bound keys give D distinct copies, so the
# working set is D times the pool; unbound keys (every request keyed under
# the first descriptor, the provenance dimension dropped) give one.
# --------------------------------------------------------------------------
@dataclass
class EvictionStream:
    chunk_tokens: int
    descriptors: list
    pool: np.ndarray          # int32[P, k * C]: the prompts
    requests_per_step: int
    budget: int               # entries (chunks)

    @property
    def P(self) -> int:
        return int(self.pool.shape[0])

    def steps_per_cycle(self) -> int:
        """Steps until every prompt has been served under every provenance once."""
        return len(self.descriptors) * self.P // self.requests_per_step

    def step(self, s: int, bound: bool) -> Batch:
        """Requests s*R .. s*R+R-1: request i is prompt i % P under provenance
        (i // P) % D (all under provenance 0 when unbound)."""
        R, P, D = self.requests_per_step, self.P, len(self.descriptors)
        first = (s * R) % P
        rows = self.pool[first:first + R]
        variant = ((s * R) // P) % D if bound else 0
        off = np.arange(R + 1, dtype=np.int64) * rows.shape[1]
        return Batch(np.ascontiguousarray(rows).reshape(-1), off, np.full(R, variant, np.uint32))


def eviction_stream(D: int, P: int = 512, k: int = 8, R: int = 64, C: int = 256, margin: float = 0.125,
                    seed: int = 5) -> EvictionStream:
    """P prompts of k chunks (C tokens, vocab 152064), R requests per step
    (R divides P), D adapters; budget = (1 + margin) * P * k entries."""
    if P % R:
        raise ValueError("R must divide P")
    rng = np.random.default_rng(seed)
    version = _hex(rng, 20)
    descs = [_desc(version=version, adapter=f"adapter-{a:02d}") for a in range(D)]
    pool = rng.integers(0, 152064, (P, k * C), dtype=np.int64).astype(np.int32)
    return EvictionStream(C, descs, pool, R, int((1 + margin) * P * k))
