#!/usr/bin/env python3
"""Benchmark: provenance-bound key derivation + longest-prefix lookup + store
of the misses on one GB300, through the libpk C-ABI.

One step = one pass of the whole hot path over one batch:
  a0  canonicalise + encode the batch's descriptors (host), SHA-256 -> d (device)
  a1  chunk digests c_i          a2  chained keys k_i
  a3  probe every key            a4  store the miss ranges
(a3 and a4 in one pass: pk_lookup_store).
Default workload: the small-block paged-cache configuration, the largest
single-GPU one (16384 requests x 2048 tokens, chunk 16, 16 descriptors, table
of 2^23 entries at load 0.6).  Without --steps, the number of timed steps is
chosen from the warm-up so that the timed region lasts at least a second.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle on the same workload

Timing: each step is bracketed by CUDA events on the launching stream; before
each step the table is restored to its seeded state (pk_table_load) and L2 is
flushed by writing a 256 MiB buffer, both outside the events.  A spin kernel
queued ahead of each step keeps the device busy while the host enqueues it,
so the events see device time only (`value`).  The `e2e` figure instead
starts on an idle stream and includes the host-to-device copy of the batch's
inputs from pinned memory, the host canonicalisation and every launch, and
the device-to-host copy of the results.
"""
from __future__ import annotations

import argparse
import gc
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tokens keyed+looked up/sec and % of SHA-256/HBM roofline (1 GB300)"
SHA_OPS_PER_COMPRESSION = 1384      # 64 rounds x 14 + 48 schedule words x 10 + 8 feed-forward
LANES_PER_SM = 128                  # 4 SM sub-partitions x 32 lanes, one instruction each per clock
L2_FLUSH_BYTES = 256 << 20
MIN_TIMED_S = 1.2                   # default timed region: long enough for several clock samples


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "sm_max_mhz": d.get("sm_max_mhz", 2070.0), "source": "measured"}
    return {"hbm_gbs": 6800.0, "sm_max_mhz": 2070.0, "source": "fallback"}


DERIVE_SOURCES = ("paper_2609_38706_gb300/csrc/pk_derive.cu", "paper_2609_38706_gb300/csrc/pk_sha256.cuh",
                  "paper_2609_38706_gb300/csrc/pk_device.cuh", "paper_2609_38706_gb300/csrc/pk_internal.h")


def derive_traffic(workload: str):
    """Cold-cache DRAM bytes of one key-derivation call, from the committed ncu
    summary of that workload (profiles/dram_traffic_<workload>.md), or None
    when there is none or the kernels changed since it was taken."""
    import hashlib
    h = hashlib.sha256()
    for f in DERIVE_SOURCES:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    fields = {}
    try:
        with open(os.path.join(ROOT, "profiles", f"dram_traffic_{workload}.md")) as fh:
            for line in fh:
                k, _, v = line.strip().partition(":")
                if v:
                    fields[k.strip()] = v.strip()
    except OSError:
        return None
    if fields.get("kernel_sources_sha256") != h.hexdigest() or fields.get("workload") != workload:
        return None
    return int(fields["derive_traffic_bytes_per_call"])


def compressions(n_keys: int, C: int) -> tuple[int, int]:
    """SHA-256 compressions per batch: chunk digests (ceil((4C + 9) / 64) each)
    and chain steps (a 96-byte message = 2 each)."""
    per_chunk = (4 * C + 9 + 63) // 64
    return n_keys * per_chunk, 2 * n_keys


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"pk_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        self.proc.wait()
        self.f.close()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for name, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(name)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def cpu_oracle_pass(wl, d_ref, table, snapshot_keys):
    """One step of the oracle on a whole batch: keys, lookup, store of the
    misses; then the inserted keys are removed again so that every pass sees
    the same table."""
    import oracle as O
    b = wl.batch
    ko, keys = O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d_ref)
    hit, slots = O.lookup(table, keys, ko)
    new_slots = np.arange(keys.shape[0], dtype=np.uint32) + (1 << 30)
    res, _ = O.store_misses(table, keys, ko, hit, new_slots)
    for i in np.nonzero(res == O.STORE_INSERTED)[0]:
        del table.map[O.prefix128(keys[i:i + 1])[0].tobytes()]
    assert len(table) == snapshot_keys
    return keys.shape[0]


def oracle_setup(wl):
    import oracle as O
    from paper_2609_38706_gb300 import workloads as W
    d_ref = O.descriptor_digests(wl.descriptors)
    pko, pkeys = O.derive_keys(wl.prior.tokens, wl.prior.tok_off, wl.chunk_tokens, wl.prior.desc_idx, d_ref)
    table = O.seed_table(O.DictTable(wl.capacity), W.seed_list(pkeys, pko, wl.prior_chunks), wl.filler,
                         wl.target_entries)
    return d_ref, table


def _hashlib_keys(task):
    """Worker of the hashlib baseline (a spawned process): the keys of requests [r0, r1)."""
    import oracle as O
    tokens, tok_off, C, desc_idx, digests, r0, r1 = task
    return O.derive_keys_hashlib(tokens, tok_off, C, desc_idx, digests, range(r0, r1)).shape[0]


def keys_rate(fn, wl, seconds: float):
    """Full-chunk tokens per second of fn() (one batch's keys per call), over about `seconds`."""
    n, t0 = 0, time.perf_counter()
    while True:
        fn()
        n += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            return wl.tokens_keyed() * n / el, n, el


def run_cpu_baseline(wl, seconds: float) -> dict:
    import multiprocessing
    import oracle as O
    d_ref, table = oracle_setup(wl)
    n0 = len(table)
    passes, t0 = 0, time.perf_counter()
    while True:
        cpu_oracle_pass(wl, d_ref, table, n0)
        passes += 1
        el = time.perf_counter() - t0
        if el >= seconds or passes >= 1000:
            break
    cores = O.max_threads()
    b = wl.batch
    part = max(seconds / 3, 1.0)
    # key derivation alone: the C oracle on one thread and on every core, and the standard library's
    # SHA-256 (OpenSSL) over a spawned process per core
    derive = lambda: O.derive_keys(b.tokens, b.tok_off, wl.chunk_tokens, b.desc_idx, d_ref)
    O.set_threads(1)
    one, n1, e1 = keys_rate(derive, wl, part)
    O.set_threads(cores)
    omp, n2, e2 = keys_rate(derive, wl, part)
    bounds = np.linspace(0, b.R, 4 * cores + 1).astype(int)
    tasks = [(b.tokens[b.tok_off[r0]:b.tok_off[r1]], b.tok_off[r0:r1 + 1] - b.tok_off[r0], wl.chunk_tokens,
              b.desc_idx[r0:r1], d_ref, 0, r1 - r0) for r0, r1 in zip(bounds[:-1], bounds[1:])]
    hl, n3, e3, why = None, 0, 0.0, ""
    try:  # every wait on the pool is bounded: a pool that cannot start reports null
        with multiprocessing.get_context("spawn").Pool(cores) as pool:
            pool.map_async(_hashlib_keys, tasks[:cores]).get(timeout=120)  # start-up outside the timing
            hl, n3, e3 = keys_rate(lambda: pool.map_async(_hashlib_keys, tasks).get(timeout=120), wl, part)
    except Exception as exc:  # (multiprocessing.TimeoutError included)
        why = f"; hashlib pool unavailable: {type(exc).__name__}"
    return {"value": wl.tokens_keyed() * passes / el, "unit": "tokens/s", "cores": cores,
            "kind": "oracle",
            "sample": f"{passes} full passes of the {wl.name} batch ({wl.batch.R} requests) in {el:.1f} s: "
                      "C FIPS 180-4 SHA-256 (OpenMP over requests) + Python dict table",
            "keys_only_tokens_per_s": {
                "c_one_thread": one, "c_all_cores": omp, "hashlib_processes": hl,
                "sample": f"key derivation of the whole batch: C {n1} passes on 1 thread ({e1:.1f} s), {n2} on "
                          f"{cores} threads ({e2:.1f} s); hashlib {n3} passes over {cores} spawned processes "
                          f"({e3:.1f} s){why}"}}


def auto_steps(iter_s: float, min_s: float = MIN_TIMED_S, lo: int = 20, hi: int = 4000) -> int:
    """Timed steps for a timed region of at least min_s, given the wall time
    of one step with its untimed preparation."""
    if iter_s <= 0:
        return lo
    return int(min(hi, max(lo, -(-min_s // iter_s))))


def critical_path(wl, derive_s: float, peaks: dict) -> dict:
    """The serial bound of key derivation: a request's chain cannot start before its first chunk digest
    and then takes 2 dependent compressions per chunk; a lone warp's compression cannot beat its
    half-rate logic/shift pipe (10 such instructions per round, one every 2 cycles, 64 rounds)."""
    C = wl.chunk_tokens
    n_max = int((np.diff(wl.batch.tok_off) // C).max()) if wl.batch.R else 0
    serial = (-(-(4 * C + 9) // 64) + 2 * n_max) if n_max else 0
    per_comp_us = 64 * 10 * 2 / peaks["sm_max_mhz"]
    bound_us = serial * per_comp_us
    return {"serial_compressions": serial, "compression_floor_us": per_comp_us, "bound_us": bound_us,
            "key_derivation_us": derive_s * 1e6, "frac": bound_us / (derive_s * 1e6) if derive_s else None,
            "basis": "first chunk digest + 2 compressions per chunk of the longest request, each at least "
                     "64 rounds x 10 logic/shift instructions x 2 cycles at the max SM clock"}


def workload_config(wl, args) -> dict:
    lens = np.diff(wl.batch.tok_off)
    return {"workload": f"{wl.name}: {wl.batch.R} requests x {int(lens.max()) if lens.size else 0} tokens, "
                        f"chunk {wl.chunk_tokens}, {len(wl.descriptors)} descriptors, table 2^{wl.capacity_log2} "
                        f"slots seeded to {wl.target_entries} entries",
            "requests": wl.batch.R, "tokens": wl.batch.n_tokens, "chunk_tokens": wl.chunk_tokens,
            "keys_per_step": wl.n_keys(), "descriptors": len(wl.descriptors), "table_slots": wl.capacity,
            "table_entries": wl.target_entries,
            "between_steps": "L2 flushed (256 MiB write) and table restored to its seeded snapshot, untimed"}


def max_over_ranks(times_ms, world: int, device=None):
    """The job's times: each the maximum over the ranks (replicas) of the
    local time; identity for one process."""
    if world <= 1:
        return [float(x) for x in times_ms]
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x) for x in times_ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t.cpu()]


def job_rate(units_per_step: float, steps: int, world: int, total_ms: float) -> float:
    """Whole-job throughput: the units all ranks processed over the slowest rank's time."""
    return units_per_step * steps * world / (total_ms / 1e3)


def run_reference(args, rank: int, world: int) -> None:
    if rank != 0:
        return
    from paper_2609_38706_gb300 import workloads as W
    import oracle as O
    wl = W.FULL_CONFIGS[args.workload]()
    d_ref, table = oracle_setup(wl)
    n0 = len(table)
    for _ in range(args.warmup):
        cpu_oracle_pass(wl, d_ref, table, n0)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        cpu_oracle_pass(wl, d_ref, table, n0)
    el = time.perf_counter() - t0
    value = wl.tokens_keyed() * args.steps / el
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": 0,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32",
            "data": "synthetic", "config": workload_config(wl, args),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": O.max_threads(), "kind": "oracle",
                             "sample": f"each step one full pass of the {wl.name} batch"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0, help="timed steps (default: a timed region of >= 1.2 s)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="pk", choices=["pk", "reference"])
    ap.add_argument("--workload", default="small_block")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if args.steps <= 0:
            args.steps = 3
        run_reference(args, rank, world)
        return

    import torch
    import torch.distributed as dist

    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_38706_gb300 import pk
    from paper_2609_38706_gb300 import workloads as W
    from paper_2609_38706_gb300.service import KeyTable

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    torch.cuda.set_stream(torch.cuda.Stream(device=dev))  # a dedicated (non-legacy) stream for all work
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    wl = W.FULL_CONFIGS[args.workload]()
    C = wl.chunk_tokens
    b = wl.batch
    stream = torch.cuda.current_stream()

    # ---- table: seeded from the prior batch by the GPU path itself ----
    kt = KeyTable(C, wl.capacity_log2, device=dev)
    d0 = kt.digests(wl.descriptors)
    pko, pkeys = kt.derive(wl.prior.tokens, wl.prior.tok_off, wl.prior.desc_idx, d0)
    pko_h = pko.cpu().numpy()
    seeds = W.seed_list(pkeys.cpu().numpy()[: int(pko_h[-1])], pko_h, wl.prior_chunks)
    kt.seed(seeds, wl.filler, wl.target_entries)
    del pkeys, pko
    snapshot = kt.save()

    # ---- resident inputs and outputs ----
    R, N_cap = b.R, b.n_tokens // C
    # The step's inputs in one pinned staging buffer, and a device buffer of the same layout (request
    # offsets, descriptor indices, tokens), so that a step moves them with one host->device copy; the
    # results likewise in one device buffer (h_r, slots, store results, output slots) and one copy back.
    def align(n, a=256):
        return (n + a - 1) // a * a
    o_desc = align(8 * (R + 1))
    o_tok = o_desc + align(4 * R)
    in_bytes = o_tok + 4 * b.n_tokens
    in_h = torch.zeros(in_bytes, dtype=torch.uint8).pin_memory()
    in_h[: 8 * (R + 1)].view(torch.int64).copy_(torch.from_numpy(b.tok_off))
    in_h[o_desc: o_desc + 4 * R].view(torch.int32).copy_(torch.from_numpy(b.desc_idx.view(np.int32)))
    in_h[o_tok:].view(torch.int32).copy_(torch.from_numpy(b.tokens))
    in_d = in_h.to(dev)

    def inputs(buf):
        return (buf[o_tok:].view(torch.int32), buf[: 8 * (R + 1)].view(torch.int64),
                buf[o_desc: o_desc + 4 * R].view(torch.int32))
    tokens_h, tok_off_h, desc_idx_h = inputs(in_h)
    tokens_d, tok_off_d, desc_idx_d = inputs(in_d)
    descs = pk.Descriptors(wl.descriptors)
    # one pinned staging buffer: D+1 int64 offsets, then the encodings; the key-derivation launch reads
    # it in place, so it is rewritten only after the previous step has completed
    off_bytes = 8 * (descs.count + 1)
    a0_h = torch.zeros(off_bytes + 256 * 1024, dtype=torch.uint8).pin_memory()
    enc_off_h = a0_h[:off_bytes].view(torch.int64)
    enc_h = a0_h[off_bytes:]
    enc_used, _ = pk.pk_descriptors_encode(descs, enc_h.numpy(), enc_off_h.numpy())
    n_enc = int(enc_used.size)
    digests_d = torch.zeros((descs.count, 32), dtype=torch.uint8, device=dev)
    key_off_d = torch.empty(R + 1, dtype=torch.int64, device=dev)
    keys_d = torch.empty((N_cap, 32), dtype=torch.uint8, device=dev)
    new_slots_d = torch.arange(N_cap, dtype=torch.int32, device=dev) + (1 << 30)
    out_d = torch.empty(R + 3 * N_cap, dtype=torch.int32, device=dev)
    out_h = torch.empty(R + 3 * N_cap, dtype=torch.int32).pin_memory()

    def outputs(buf):
        return buf[:R], buf[R: R + N_cap], buf[R + N_cap: R + 2 * N_cap], buf[R + 2 * N_cap:]
    hit_d, slots_d, result_d, slot_out_d = outputs(out_d)
    hit_h, slots_h, result_h, slot_out_h = outputs(out_h)
    status = kt.status
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    ctx = kt.ctx

    def core(ev=None):
        pk.pk_descriptors_encode(descs, enc_h.numpy(), enc_off_h.numpy())      # a0, host: canonicalise + enc
        if ev: ev[1].record(stream)
        # a0 (descriptor SHA-256), a1 (chunk digests), a2 (chain) in one call.  The encodings are read by
        # the kernel straight from the pinned staging buffer (host memory is device-addressable over
        # NVLink-C2C), so no copy is enqueued for them.
        pk.pk_derive_keys_enc(ctx, tokens_d, tok_off_d, desc_idx_d, enc_h[:n_enc], enc_off_h, digests_d, key_off_d,
                              keys_d, status)
        if ev: ev[2].record(stream)
        # a3 (lookup as of the start of the call) and a4 (store of the miss ranges) in one pass
        pk.pk_lookup_store(ctx, keys_d, new_slots_d, key_off_d, hit_d, slots_d, result_d, slot_out_d, status)

    def between_steps():
        kt.load(snapshot)
        flush.fill_(1)

    # The spin kernel ahead of each step (outside its events) keeps the device busy while the host enqueues
    # the step: about 1 ms, so that a short host pause inside the enqueue (a driver query of the clock
    # sampler, say) does not leave the device idle between the step's events.
    spin_cycles = int(1e-3 * 2.0e9)
    n_keys = wl.n_keys()

    # ---- warm-up, then timed device-resident steps ----
    t_warm = time.perf_counter()
    for _ in range(args.warmup):
        between_steps()
        torch.cuda._sleep(spin_cycles)
        core()
        torch.cuda.synchronize()
    iter_s = (time.perf_counter() - t_warm) / args.warmup
    if args.steps <= 0:  # a timed region of at least MIN_TIMED_S, the same on every rank
        args.steps = int(max_over_ranks([auto_steps(iter_s)], world, dev)[0])
    if kt.take_status() != 0:
        raise RuntimeError("device status after warm-up")
    hit_ref = hit_d.cpu().numpy().copy()
    inserted = kt.entries() - wl.target_entries  # keys one step inserts (the table is restored between steps)

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    # Only a start and an end event per timed step: an event recorded between two kernels also ends the
    # programmatic overlap of the second with the first.
    step_ms = []
    gc.collect()
    gc.disable()  # no collection pause while a step is being enqueued
    for _ in range(args.steps):
        between_steps()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(spin_cycles)
        e0.record(stream)
        core()
        e1.record(stream)
        torch.cuda.synchronize()
        step_ms.append(e0.elapsed_time(e1))
    gc.enable()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    if kt.take_status() != 0:
        raise RuntimeError("device status after timed steps")
    if not np.array_equal(hit_d.cpu().numpy(), hit_ref):
        raise RuntimeError("hit lengths changed between steps")

    # ---- phase breakdown: extra steps with events between the phases (not part of `value`) ----
    derive_ms, table_ms, a0_ms = [], [], []
    for _ in range(max(3, min(args.steps, 10))):
        between_steps()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        torch.cuda._sleep(spin_cycles)
        ev[0].record(stream)
        core(ev)
        ev[3].record(stream)
        torch.cuda.synchronize()
        a0_ms.append(ev[0].elapsed_time(ev[1]))
        derive_ms.append(ev[1].elapsed_time(ev[2]))
        table_ms.append(ev[2].elapsed_time(ev[3]))

    # ---- e2e: host buffers, host->device transfer inside the timed region ----
    # "in_place": the kernels read tokens, offsets, descriptor indices and encodings straight from the
    # pinned host buffers (device-addressable over NVLink-C2C), so the transfer overlaps the hashing;
    # "staged": explicit pinned->device copies first.  Both end with device->host copies of the results.
    def e2e_step(in_place: bool):
        if in_place:
            pk.pk_descriptors_encode(descs, enc_h.numpy(), enc_off_h.numpy())
            pk.pk_derive_keys_enc(ctx, tokens_h, tok_off_h, desc_idx_h, enc_h[:n_enc], enc_off_h, digests_d,
                                  key_off_d, keys_d, status)
            pk.pk_lookup_store(ctx, keys_d, new_slots_d, key_off_d, hit_d, slots_d, result_d, slot_out_d,
                               status)
        else:
            in_d.copy_(in_h, non_blocking=True)
            core()
        out_h.copy_(out_d, non_blocking=True)

    e2e_ms = {True: [], False: []}
    for in_place in (True, False):
        for i in range(args.warmup + args.steps):
            between_steps()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            e2e_step(in_place)
            e1.record(stream)
            torch.cuda.synchronize()
            if i >= args.warmup:
                e2e_ms[in_place].append(e0.elapsed_time(e1))
    if kt.take_status() != 0:
        raise RuntimeError("device status after e2e steps")
    if not np.array_equal(hit_h.numpy(), hit_ref):
        raise RuntimeError("e2e hit lengths differ from the device-resident run")
    h2d = in_bytes + off_bytes + n_enc
    d2h = out_h.numel() * 4

    total_ms = float(np.sum(step_ms))
    e2e_total = float(np.sum(e2e_ms[False]))
    e2e_inplace_total = float(np.sum(e2e_ms[True]))
    total_ms, e2e_total, e2e_inplace_total = max_over_ranks([total_ms, e2e_total, e2e_inplace_total], world, dev)
    tokens_per_step = wl.tokens_keyed()
    value = job_rate(tokens_per_step, args.steps, world, total_ms)
    e2e_value = job_rate(tokens_per_step, args.steps, world, e2e_total)

    peaks = load_peaks()
    c_dig, c_chain = compressions(n_keys, C)
    derive_s = float(np.mean(derive_ms)) / 1e3
    alu_peak = sms * LANES_PER_SM * peaks["sm_max_mhz"] * 1e6 / 1e12           # Tops/s, issue-rate ceiling
    # the logic/shift pipe takes 16 lanes per sub-partition per clock and SHA-256 with funnel-shift
    # rotations needs 1024 of its operations per compression (6 SHF + 4 LOP3 per round, 6 + 2 per
    # schedule word): the ceiling for this formulation, in the same 1384-op units
    alu_pipe_peak = sms * 64 * peaks["sm_max_mhz"] * 1e6 / 1024 * SHA_OPS_PER_COMPRESSION / 1e12
    achieved = (c_dig + c_chain) * SHA_OPS_PER_COMPRESSION / derive_s / 1e12
    table_s = float(np.mean(table_ms)) / 1e3
    # per key: 16 B key + one 32 B entry sector + 4 B new slot + 12 B of outputs (lookup slot, result,
    # output slot); per inserted key one 32 B entry sector written; 4 B (h_r) per request
    probe_bytes = n_keys * (16 + 32 + 4 + 12) + inserted * 32 + R * 4
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps,
        "step_ms_min_median_max": [float(np.min(step_ms)), float(np.median(step_ms)), float(np.max(step_ms))],
        "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u32", "data": "synthetic",
        "config": workload_config(wl, args),
        "lookups_per_s": job_rate(n_keys, args.steps, world, total_ms),
        "requests_per_s": job_rate(R, args.steps, world, total_ms),
        "phase_ms": {"a0_host": float(np.mean(a0_ms)), "descriptors_and_keys": float(np.mean(derive_ms)),
                     "lookup_and_store": float(np.mean(table_ms)),
                     "note": "separate steps with events between the phases (each event also ends the "
                             "overlap of the next launch with the previous one)"},
        "inserted_per_step": inserted,
        "roofline": {"bound": "alu",
                     "kernel": "pk_derive_keys_enc (chunk offsets; chunk + descriptor digests; chain)",
                     "achieved": achieved, "peak": alu_peak, "unit": "Tops/s", "frac": achieved / alu_peak,
                     "traffic": derive_traffic(args.workload),
                     "algorithmic_bytes": wl.batch.n_tokens * 4 + n_keys * 32,
                     "alu_pipe_peak": alu_pipe_peak,
                     "peak_basis": f"{sms} SMs (device query) x {LANES_PER_SM} int32 lanes x {peaks['sm_max_mhz']:.0f} MHz "
                                   f"(issue-rate ceiling); {SHA_OPS_PER_COMPRESSION} ops per compression, "
                                   f"{c_dig + c_chain} compressions per launch"},
        "probe_roofline": {"bound": "hbm", "kernel": "pk_lookup_store (probe + claim; finalize)",
                           "achieved": probe_bytes / table_s / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                           "frac": probe_bytes / table_s / 1e9 / peaks["hbm_gbs"],
                           "bytes_basis": "per key 16 B key + one 32 B entry sector + 4 B new slot + 12 B "
                                          "outputs; 32 B per inserted key; 4 B per request",
                           "peak_source": peaks["source"]},
        "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_total / args.steps,
                "h2d": "one pinned host -> device copy of tokens, request offsets and descriptor indices "
                       "(descriptor encodings read in place); one copy of the results back",
                "in_place_reads": {"value": job_rate(tokens_per_step, args.steps, world, e2e_inplace_total),
                                   "ms_per_step": e2e_inplace_total / args.steps,
                                   "note": "all inputs read by the kernels from pinned host memory"}},
        # per step: chunk offsets, chunk+descriptor digests, chain; lookup-and-store (one kernel of
        # request warps, or per key + per-request tail for few long requests); finalize
        "critical_path": critical_path(wl, derive_s, peaks),
        "gpu_launches": (3 + (1 if (R >= 1024 or N_cap <= 64 * R) else 2) + 1) * args.steps,
        "clocks": clk,
    }
    # Store-side omission test (comparison step, pk_compare_pages): 16,384 joined pages of 16 KiB against a
    # reference set, 1/8 of them absent and 1/4 differing in one byte; HBM-bound.  The 512 MiB of pages are
    # larger than L2, so no flush between repetitions (a flush's dirty lines would be written back during
    # the next read).
    n_pg, pg_bytes = 16384, 16384
    gen = torch.Generator(device=dev).manual_seed(7)
    ref_pages = torch.randint(0, 256, (n_pg, pg_bytes), dtype=torch.uint8, device=dev, generator=gen)
    perm = torch.randperm(n_pg, device=dev, generator=gen)
    pages = ref_pages[perm].clone()
    pages[: n_pg // 4, pg_bytes // 2] ^= 1
    pg_slots = perm.to(torch.int32)
    pg_slots[n_pg - n_pg // 8:] = -1                        # PK_NO_SLOT
    verdict = torch.empty(n_pg, dtype=torch.int32, device=dev)
    counts = torch.zeros(3, dtype=torch.int64, device=dev)
    cmp_ms = []
    for it in range(8):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        pk.pk_compare_pages(pg_slots, pages, ref_pages, verdict, counts, status)
        e1.record(stream)
        torch.cuda.synchronize()
        if it >= 3:
            cmp_ms.append(e0.elapsed_time(e1))
    if kt.take_status() != 0 or counts.tolist() != [8 * (n_pg // 8), 8 * (n_pg - n_pg // 8 - n_pg // 4),
                                                     8 * (n_pg // 4)]:
        raise RuntimeError("page comparison counts")
    present = n_pg - n_pg // 8
    cmp_bytes = 2 * present * pg_bytes + n_pg * 8
    cmp_gbs = cmp_bytes / (float(np.mean(cmp_ms)) / 1e3) / 1e9
    del ref_pages, pages

    # Connector key strings (pk_key_strings): the step's keys as 150-byte rows (prefix, 22 base64
    # characters, zero fill), and 16M random keys (2.4 GB of rows) for the HBM roofline.
    ks_width = 150
    ks_prefix = ("vllm@" + pk.pk_model_tag(wl.descriptors[0]) + "@1@0@").encode()

    def key_strings_us(keys, n, reps=8):
        rows = torch.empty((n, ks_width), dtype=torch.uint8, device=dev)
        times = []
        for it in range(reps + 3):
            flush.fill_(1)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            pk.pk_key_strings(keys, ks_prefix, ks_width, rows, n=n)
            e1.record(stream)
            torch.cuda.synchronize()
            if it >= 3:
                times.append(e0.elapsed_time(e1) * 1e3)
        del rows
        return float(np.mean(times))
    ks_step_us = key_strings_us(keys_d, n_keys)
    n_big = 16 << 20
    big_keys = torch.randint(0, 256, (n_big, 32), dtype=torch.uint8, device=dev, generator=gen)
    ks_big_us = key_strings_us(big_keys, n_big, reps=5)
    del big_keys
    ks_bytes = n_big * (16 + ks_width)
    ks_gbs = ks_bytes / (ks_big_us * 1e-6) / 1e9
    line["key_strings"] = {
        "step_keys": n_keys, "step_us": ks_step_us, "width": ks_width, "prefix_bytes": len(ks_prefix),
        "roofline": {"bound": "hbm", "kernel": "pk_key_strings", "keys": n_big, "us": ks_big_us,
                     "achieved": ks_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": ks_gbs / peaks["hbm_gbs"],
                     "bytes_basis": f"16 B key prefix read + {ks_width} B row written per key",
                     "peak_source": peaks["source"]}}

    # Eviction under a fixed budget (pk_evict).  (1) The kernel on a 2^22-entry table holding 2M entries
    # (stamps from one list-mode store), evicting to 1M: restored and L2-flushed before each repetition.
    # (2) The call within the budget (returns at once).  (3) The thrashing of Sec. 6.5 on the key path:
    # one prompt pool served under D adapters in turn, budget about one copy of the pool, evicting after
    # every step; bound keys (one copy per adapter) against unbound keys (one copy in all).
    ev_log2, ev_n = 22, 2 << 20
    kt_ev = KeyTable(16, ev_log2, device=dev)
    kt_ev.attach_stamps()
    ev_keys = torch.randint(0, 256, (ev_n, 32), dtype=torch.uint8, device=dev, generator=gen)
    ev_keys[:, 0] |= 1
    kt_ev.store(ev_keys, torch.arange(ev_n, dtype=torch.int32, device=dev))
    del ev_keys
    torch.cuda.synchronize()
    if kt_ev.take_status() != 0:
        raise RuntimeError("eviction table fill")
    ev_entries = kt_ev.entries()
    ev_snap, ev_stamps = kt_ev.save(), kt_ev.stamps.clone()

    def evict_us(budget, keep, reps):
        times, n_out = [], 0
        for it in range(reps + 2):
            kt_ev.load(ev_snap)
            kt_ev.stamps.copy_(ev_stamps)
            flush.fill_(1)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            _, n_ev = kt_ev.evict(budget, keep)
            e1.record(stream)
            torch.cuda.synchronize()
            if it >= 2:
                times.append(e0.elapsed_time(e1) * 1e3)
            n_out = int(n_ev.item())
        if kt_ev.take_status() != 0:
            raise RuntimeError("evict status")
        return float(np.mean(times)), n_out
    ev_keep = ev_entries // 2
    ev_us, ev_removed = evict_us(ev_entries - 1, ev_keep, 5)
    if ev_removed != ev_entries - ev_keep or kt_ev.entries() != ev_keep:
        raise RuntimeError("eviction count")
    idle_us, idle_removed = evict_us(ev_entries, ev_keep, 10)
    kt_ev.close()
    del kt_ev, ev_snap, ev_stamps
    # bytes: the gather reads one 32 B entry sector per table entry and 8 B of stamp per entry held; the
    # compaction rewrites the removed entries (32 B + 8 B of stamp each)
    ev_bytes = (1 << ev_log2) * 32 + ev_entries * 8 + ev_removed * 40
    thrash = []
    for D in (1, 2, 4):
        for bound in ((True,) if D == 1 else (True, False)):
            es = W.eviction_stream(D)
            kts = KeyTable(es.chunk_tokens, 14, device=dev)
            kts.attach_stamps()
            dg = kts.digests(es.descriptors)
            pool_d = torch.from_numpy(es.pool).to(dev)
            Rs, kch = es.requests_per_step, es.pool.shape[1] // es.chunk_tokens
            tok_off_s = torch.arange(Rs + 1, dtype=torch.int64, device=dev) * es.pool.shape[1]
            key_off_s = torch.empty(Rs + 1, dtype=torch.int64, device=dev)
            keys_s = torch.empty((Rs * kch, 32), dtype=torch.uint8, device=dev)
            hit_s = torch.empty(Rs, dtype=torch.int32, device=dev)
            outs = torch.empty((3, Rs * kch), dtype=torch.int32, device=dev)
            cyc = es.steps_per_cycle()
            hits = chunks = evicted = 0
            st_us = []
            for s in range(3 * cyc):
                bt = es.step(s, bound)
                first = (s * Rs) % es.P
                toks = pool_d[first:first + Rs].reshape(-1)
                didx = torch.full((Rs,), int(bt.desc_idx[0]), dtype=torch.int32, device=dev)
                slots_new = torch.arange(Rs * kch, dtype=torch.int32, device=dev) + s * Rs * kch
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                pk.pk_derive_keys(kts.ctx, toks, tok_off_s, didx, dg, key_off_s, keys_s, kts.status)
                pk.pk_lookup_store(kts.ctx, keys_s, slots_new, key_off_s, hit_s, outs[0], outs[1], outs[2],
                                   kts.status)
                _, n_ev = kts.evict(es.budget, es.budget)
                e1.record(stream)
                torch.cuda.synchronize()
                if s >= cyc:  # after the first cycle
                    st_us.append(e0.elapsed_time(e1) * 1e3)
                    hits += int(hit_s.sum().item())
                    chunks += Rs * kch
                    evicted += int(n_ev.item())
            if kts.take_status() != 0:
                raise RuntimeError("thrash status")
            thrash.append({"D": D, "bound": bound, "hit_rate": hits / chunks, "step_us": float(np.mean(st_us)),
                           "evicted_per_step": evicted / len(st_us), "working_set_chunks": (D if bound else 1)
                           * es.P * kch, "budget_chunks": es.budget})
            kts.close()
    line["eviction"] = {
        "evict_us": ev_us, "table_entries": ev_entries, "removed": ev_removed, "capacity": 1 << ev_log2,
        "within_budget_us": idle_us,
        "achieved_GBps": ev_bytes / (ev_us * 1e-6) / 1e9, "peak_GBps": peaks["hbm_gbs"],
        "frac": ev_bytes / (ev_us * 1e-6) / 1e9 / peaks["hbm_gbs"],
        "bytes_basis": "32 B entry sector per table entry + 8 B stamp per entry held + 40 B per removed entry",
        "thrash": thrash,
        "thrash_setup": "512 prompts x 8 chunks of 256 tokens, 64 requests per step, prompt i % 512 under "
                        "adapter (i // 512) % D, budget 4608 entries (1.125 copies), evict after each step; "
                        "hit rate and step time (derive + lookup-and-store + evict) over cycles 2-3",
        "paper": "vLLM, bound: TTFT 0.024 -> 0.065 s, 42 -> 15 req/s once capacity is exceeded; unbound flat"}

    # Content identity (pk_content_digest, the SHA-256 tree): a 40 MB adapter as 16 tensors, and a 1 GiB
    # checkpoint buffer; random bytes generated on the device.
    def content_us(sizes, reps=5, batched=True):
        bufs = [torch.randint(0, 256, (n,), dtype=torch.uint8, device=dev, generator=gen) for n in sizes]
        scr = torch.empty(pk.pk_content_scratch_bytes_batch(sizes), dtype=torch.uint8, device=dev)
        tops = torch.empty((len(sizes), 32), dtype=torch.uint8, device=dev)
        times = []
        for it in range(reps + 2):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            if batched:  # every tree level of all the tensors in one launch
                pk.pk_content_digests(bufs, scr, tops)
            else:
                for j, bf in enumerate(bufs):
                    pk.pk_content_digest(bf, scr, tops[j])
            e1.record(stream)
            torch.cuda.synchronize()
            if it >= 2:
                times.append(e0.elapsed_time(e1) * 1e3)
        del bufs
        return float(np.mean(times))

    def tree_compressions(n):
        total, m = 0, max(1, -(-n // 1024))
        while True:
            total += 17 * m
            if m == 1:
                return total
            m = max(1, -(-(32 * m) // 1024))
    adapter_sizes = [40 * 10**6 // 16] * 16
    ckpt_sizes = [1 << 30]
    ad_us, ck_us = content_us(adapter_sizes), content_us(ckpt_sizes, reps=3)
    ad_single_us = content_us(adapter_sizes, batched=False)
    ck_comp = tree_compressions(ckpt_sizes[0])
    line["content_identity"] = {
        "adapter_40MB_us": ad_us, "adapter_40MB_one_call_per_tensor_us": ad_single_us, "checkpoint_1GiB_us": ck_us,
        "checkpoint_GBps": ckpt_sizes[0] / (ck_us * 1e-6) / 1e9,
        "checkpoint_G_compressions_per_s": ck_comp / (ck_us * 1e-6) / 1e9,
        "alu_pipe_peak_G_compressions_per_s": sms * 64 * peaks["sm_max_mhz"] * 1e6 / 1024 / 1e9,
        "paper_host": "adapter 40 MB: 1.06 s cold, 0.060 s warm; 0.5B checkpoint content hash: 1.35 s"}

    # Two-level variant (request- and worker-level digests): the host cost of one request's digest under a
    # worker digest computed once, through the C ABI over the batch's R requests.
    req_descs = pk.Descriptors([wl.descriptors[int(i)] for i in b.desc_idx])
    worker = pk.pk_worker_digest(wl.descriptors[0])
    reps = 5
    t0 = time.perf_counter()
    for _ in range(reps):
        pk.pk_request_digests(worker, req_descs)
    line["two_level_request_digest_us"] = (time.perf_counter() - t0) / (reps * R) * 1e6
    line["omission_check_roofline"] = {
        "bound": "hbm", "kernel": "pk_compare_pages", "achieved": cmp_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
        "frac": cmp_gbs / peaks["hbm_gbs"], "us": float(np.mean(cmp_ms)) * 1e3,
        "bytes_basis": f"{n_pg} joined pages of {pg_bytes} B ({present} present, each read twice) + 8 B per key",
        "peak_source": peaks["source"]}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = run_cpu_baseline(wl, args.cpu_seconds)
    if rank == 0:
        print(json.dumps(line), flush=True)
    kt.close()
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
