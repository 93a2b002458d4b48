"""Convenience layer over the C-ABI: a device-resident key table plus
per-batch buffers, all allocated with PyTorch, every step run by libpk.

    kt = KeyTable(chunk_tokens=256, capacity_log2=20)
    d = kt.digests(descriptors)                  # a0: canonicalise + enc (host), SHA-256 (device)
    key_off, keys = kt.derive(tokens, tok_off, desc_idx, d)      # a1 + a2
    hit, slots = kt.lookup(keys, key_off)                        # a3
    result, slot_out = kt.store(keys, new_slots, key_off, hit)   # a4 (the misses)
"""
from __future__ import annotations

from typing import Optional

import numpy as np
import torch

from . import pk


_NP_SIGNED = {torch.int32: np.int32, torch.int64: np.int64, torch.uint8: np.uint8}


def _dev(x, dtype, device) -> torch.Tensor:
    """Host array or tensor -> contiguous device tensor of ``dtype``; unsigned
    host arrays of the same width are reinterpreted, not converted."""
    if isinstance(x, torch.Tensor):
        return x.to(device=device, dtype=dtype).contiguous()
    a = np.ascontiguousarray(x)
    want = np.dtype(_NP_SIGNED[dtype])
    a = a.view(want) if a.dtype.itemsize == want.itemsize and a.dtype.kind in "ui" else a.astype(want)
    return torch.from_numpy(a).to(device=device)


class KeyTable:
    def __init__(self, chunk_tokens: int, capacity_log2: int, max_probe: int = 0, device="cuda",
                 stream: Optional[torch.cuda.Stream] = None):
        self.device = torch.device(device)
        self.stream = stream
        self.chunk_tokens = int(chunk_tokens)
        self.capacity_log2 = int(capacity_log2)
        nbytes = pk.pk_table_bytes(capacity_log2)
        if nbytes == 0:
            raise pk.PKError(pk.PK_ERR_CAPACITY, "KeyTable")
        self.table = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        self.status = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.ctx = pk.pk_init(self.table, chunk_tokens, capacity_log2, max_probe, stream)

    # -- lifecycle ---------------------------------------------------------
    def close(self):
        if self.ctx:
            torch.cuda.synchronize(self.device)
            pk.pk_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def entries(self) -> int:
        return pk.pk_entries(self.ctx, self.stream)

    def save(self, dst: Optional[torch.Tensor] = None) -> torch.Tensor:
        """Checkpoint the table (device tensor unless ``dst`` is given)."""
        if dst is None:
            dst = torch.empty(self.table.numel() + 64, dtype=torch.uint8, device=self.device)
        pk.pk_table_save(self.ctx, dst, self.stream)
        return dst

    def load(self, src: torch.Tensor) -> None:
        pk.pk_table_load(self.ctx, src, self.stream)

    def take_status(self) -> int:
        """Read and clear the device status word (synchronises)."""
        v = int(self.status.item())
        self.status.zero_()
        return v

    def check(self, where: str = "device") -> None:
        v = self.take_status()
        if v != pk.PK_OK:
            raise pk.PKError(v, where)

    # -- steps -------------------------------------------------------------
    def digests(self, descriptors) -> torch.Tensor:
        enc, off = pk.pk_descriptors_encode(descriptors)
        D = off.size - 1
        enc_d = _dev(enc if enc.size else np.zeros(1, np.uint8), torch.uint8, self.device)
        off_d = _dev(off, torch.int64, self.device)
        out = torch.zeros((max(D, 1), 32), dtype=torch.uint8, device=self.device)
        pk.pk_digest_descriptors(self.ctx, enc_d[: enc.size], off_d, out, self.status, self.stream)
        return out[:D]

    def derive(self, tokens, tok_off, desc_idx, digests):
        tokens = _dev(tokens, torch.int32, self.device)
        tok_off = _dev(tok_off, torch.int64, self.device)
        desc_idx = _dev(desc_idx, torch.int32, self.device)
        R = tok_off.numel() - 1
        cap = tokens.numel() // self.chunk_tokens
        key_off = torch.empty(R + 1, dtype=torch.int64, device=self.device)
        keys = torch.empty((max(cap, 0), 32), dtype=torch.uint8, device=self.device)
        pk.pk_derive_keys(self.ctx, tokens, tok_off, desc_idx, digests, key_off, keys, self.status, self.stream)
        return key_off, keys

    def derive_enc(self, tokens, tok_off, desc_idx, descriptors):
        """Descriptor digests and keys in one call (pk_derive_keys_enc)."""
        enc, off = pk.pk_descriptors_encode(descriptors)
        D = off.size - 1
        enc_d = _dev(enc if enc.size else np.zeros(1, np.uint8), torch.uint8, self.device)[: enc.size]
        off_d = _dev(off, torch.int64, self.device)
        digests = torch.zeros((max(D, 1), 32), dtype=torch.uint8, device=self.device)[:D]
        tokens = _dev(tokens, torch.int32, self.device)
        tok_off = _dev(tok_off, torch.int64, self.device)
        desc_idx = _dev(desc_idx, torch.int32, self.device)
        R = tok_off.numel() - 1
        cap = tokens.numel() // self.chunk_tokens
        key_off = torch.empty(R + 1, dtype=torch.int64, device=self.device)
        keys = torch.empty((max(cap, 0), 32), dtype=torch.uint8, device=self.device)
        pk.pk_derive_keys_enc(self.ctx, tokens, tok_off, desc_idx, enc_d, off_d, digests, key_off, keys,
                              self.status, self.stream)
        return digests, key_off, keys

    def lookup(self, keys, key_off):
        R = key_off.numel() - 1
        hit = torch.empty(R, dtype=torch.int32, device=self.device)
        slots = torch.empty(keys.shape[0], dtype=torch.int32, device=self.device)
        pk.pk_lookup(self.ctx, keys, key_off, hit, slots, self.status, self.stream)
        return hit, slots

    def store(self, keys, slots, key_off=None, hit=None):
        """List mode (key_off is None) or miss-range mode (key_off and hit)."""
        if keys.shape[1] == 16:  # widen 16-byte prefixes to the 32-byte key stride
            k = torch.zeros((keys.shape[0], 32), dtype=torch.uint8, device=self.device)
            k[:, :16] = _dev(keys, torch.uint8, self.device)
            keys = k
        else:
            keys = _dev(keys, torch.uint8, self.device)
        slots = _dev(slots if isinstance(slots, torch.Tensor) else np.asarray(slots, np.uint32), torch.int32,
                     self.device)
        n = keys.shape[0]
        result = torch.empty(n, dtype=torch.int32, device=self.device)
        slot_out = torch.empty(n, dtype=torch.int32, device=self.device)
        pk.pk_store(self.ctx, keys, slots, result, slot_out, self.status, key_off, hit, self.stream)
        return result, slot_out

    def lookup_store(self, keys, key_off, new_slots):
        """lookup followed by store of the miss ranges, in one pass: returns
        (hit, slots, result, slot_out) as the two calls would."""
        R = key_off.numel() - 1
        n = keys.shape[0]
        new_slots = _dev(new_slots if isinstance(new_slots, torch.Tensor) else np.asarray(new_slots, np.uint32),
                         torch.int32, self.device)
        hit = torch.empty(R, dtype=torch.int32, device=self.device)
        slots = torch.empty(n, dtype=torch.int32, device=self.device)
        result = torch.empty(n, dtype=torch.int32, device=self.device)
        slot_out = torch.empty(n, dtype=torch.int32, device=self.device)
        pk.pk_lookup_store(self.ctx, keys, new_slots, key_off, hit, slots, result, slot_out, self.status,
                           self.stream)
        return hit, slots, result, slot_out

    def derive_lookup_store(self, tokens, tok_off, desc_idx, descriptors, new_slots):
        """The whole hot path in one call (pk_derive_lookup_store): returns
        (digests, key_off, keys, hit, slots, result, slot_out)."""
        enc, off = pk.pk_descriptors_encode(descriptors)
        D = off.size - 1
        enc_d = _dev(enc if enc.size else np.zeros(1, np.uint8), torch.uint8, self.device)[: enc.size]
        off_d = _dev(off, torch.int64, self.device)
        digests = torch.zeros((max(D, 1), 32), dtype=torch.uint8, device=self.device)[:D]
        tokens = _dev(tokens, torch.int32, self.device)
        tok_off = _dev(tok_off, torch.int64, self.device)
        desc_idx = _dev(desc_idx, torch.int32, self.device)
        R = tok_off.numel() - 1
        cap = tokens.numel() // self.chunk_tokens
        key_off = torch.empty(R + 1, dtype=torch.int64, device=self.device)
        keys = torch.empty((max(cap, 0), 32), dtype=torch.uint8, device=self.device)
        new_slots = _dev(new_slots if isinstance(new_slots, torch.Tensor) else np.asarray(new_slots, np.uint32),
                         torch.int32, self.device)
        hit = torch.empty(R, dtype=torch.int32, device=self.device)
        slots = torch.empty(max(cap, 0), dtype=torch.int32, device=self.device)
        result = torch.empty(max(cap, 0), dtype=torch.int32, device=self.device)
        slot_out = torch.empty(max(cap, 0), dtype=torch.int32, device=self.device)
        pk.pk_derive_lookup_store(self.ctx, tokens, tok_off, desc_idx, enc_d, off_d, digests, key_off, keys, new_slots,
                                  hit, slots, result, slot_out, self.status, self.stream)
        return digests, key_off, keys, hit, slots, result, slot_out

    # -- budget mode (eviction under a fixed budget) -------------------------
    def attach_stamps(self) -> torch.Tensor:
        """Turn budget mode on: a zeroed last-use stamp per entry, and the
        scratch and output buffers of evict()."""
        cap = 1 << self.capacity_log2
        self.stamps = torch.empty(pk.pk_stamps_bytes(self.capacity_log2) // 8, dtype=torch.int64, device=self.device)
        pk.pk_attach_stamps(self.ctx, self.stamps, self.stream)
        self.evict_scratch = torch.empty(pk.pk_evict_scratch_bytes(self.capacity_log2), dtype=torch.uint8,
                                         device=self.device)
        self.evicted = torch.empty(cap, dtype=torch.int32, device=self.device)
        self.n_evicted = torch.zeros(1, dtype=torch.int64, device=self.device)
        return self.stamps

    def evict(self, budget: int, keep: int):
        """Enqueue pk_evict; returns (evicted slots buffer, count tensor),
        valid up to the count once the stream has run."""
        pk.pk_evict(self.ctx, budget, keep, self.evict_scratch, self.evicted, self.n_evicted, self.status,
                    self.stream)
        return self.evicted, self.n_evicted

    def seed(self, seed_keys, filler, target_entries: int) -> int:
        """Pre-fill: seed keys in order (slot = list index), then filler keys
        (continuing the index) until the table holds target_entries entries."""
        n_seed = int(seed_keys.shape[0])
        if n_seed:
            self.store(seed_keys, np.arange(n_seed, dtype=np.uint32))
        need = target_entries - self.entries()
        if need > 0:
            self.store(filler[:need], np.arange(n_seed, n_seed + need, dtype=np.uint32))
        self.check("seed")
        return self.entries()


def u32(t: torch.Tensor) -> np.ndarray:
    """int32 device tensor holding uint32 values -> numpy uint32."""
    return t.cpu().numpy().view(np.uint32)
