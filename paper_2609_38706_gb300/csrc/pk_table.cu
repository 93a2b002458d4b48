// pk_table.cu -- GPU-resident key table: lookup and store kernels (sm_103a).
//
// The shared store of the paper (Sec. 2.1) reduced to its key index: an
// open-addressing table of 2^b entries of 32 bytes (one DRAM sector each),
// keyed by the first 16 bytes of k_i (the 128-bit digest of Sec. 5.3) and
// holding the uint32 slot of the chunk's cached state.  Home position =
// (first 8 key bytes read as a little-endian integer) mod 2^b; linear probing
// with wrap-around; the all-zero key marks an empty entry.  At most
// capacity - 1 entries are ever stored, so every probe meets an empty entry;
// every probe loop is additionally bounded by max_probe.
//
// Lookup (Sec. 2.1: on a local miss the connector queries the store) reads
// the table only.  Store ("a miss computes and writes new state") inserts
// missing keys with a 128-bit compare-and-swap on the key, and resolves
// duplicates within one call to the lowest entry index in a second kernel, so
// that the result equals processing the entries one at a time in order.
#include <cuda_runtime.h>

#include "pk_device.cuh"
#include "pk_internal.h"

#include <mutex>

namespace {

using pk::set_status;

__device__ __forceinline__ bool is_zero(const uint4 &v) { return (v.x | v.y | v.z | v.w) == 0u; }
__device__ __forceinline__ bool same(const uint4 &a, const uint4 &b) {
    return ((a.x ^ b.x) | (a.y ^ b.y) | (a.z ^ b.z) | (a.w ^ b.w)) == 0u;
}
__device__ __forceinline__ uint64_t home_of(const uint4 &k) {
    return ((uint64_t)k.y << 32) | k.x;  // bytes 0..7, little-endian
}

// Loads that observe concurrent writes of the same kernel.
__device__ __forceinline__ uint4 ld_volatile_v4(const uint32_t *p) {
    uint4 v;
    asm volatile("ld.volatile.global.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}
__device__ __forceinline__ unsigned long long ld_volatile_u64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.volatile.global.u64 %0, [%1];" : "=l"(v) : "l"(p));
    return v;
}

// Entries are examined in windows of up to kWin consecutive entries (one
// 128-byte line, aligned): the keys of a window are loaded together, so a
// probe sequence costs one memory round trip per window instead of one per
// entry.  The examination order is still home, home+1, ... as in plain
// linear probing.
constexpr uint32_t kWin = 4;

// ---------------------------------------------------------------------------
// Lookup of one key: its slot, or PK_NO_SLOT.  Returns false if the probe
// sequence reached max_probe without an answer.
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool probe(const pk_entry *__restrict__ table, uint64_t mask, uint32_t max_probe,
                                      const uint4 &key, uint32_t &slot) {
    slot = PK_NO_SLOT;
    if (is_zero(key)) return true;  // the empty marker is never stored
    const uint32_t win = mask + 1 < kWin ? (uint32_t)(mask + 1) : kWin;
    const uint64_t pos = home_of(key) & mask;
    uint64_t base = pos & ~(uint64_t)(win - 1);
    uint32_t j0 = (uint32_t)(pos - base);
    uint32_t probed = 0;
    bool done = false;
    while (!done && probed < max_probe) {
        const pk_entry *grp = table + base;
        uint4 v[kWin];
#pragma unroll
        for (uint32_t u = 0; u < kWin; ++u)
            if (u < win) v[u] = __ldg(reinterpret_cast<const uint4 *>(grp[u].k));
#pragma unroll
        for (uint32_t u = 0; u < kWin; ++u) {
            if (u < win && u >= j0 && !done && probed < max_probe) {
                ++probed;
                if (same(v[u], key)) {
                    slot = __ldg(&grp[u].slot);
                    done = true;
                } else if (is_zero(v[u])) {
                    done = true;
                }
            }
        }
        base = (base + win) & mask;
        j0 = 0;
    }
    return done;
}

// One warp per request: every key's slot, and h_r = index of the first miss
// (ballot over each group of 32 keys).  For batches of many short requests.
__global__ void __launch_bounds__(256)
k_lookup_req(const pk_entry *__restrict__ table, uint64_t mask, uint32_t max_probe,
             const uint8_t *__restrict__ keys, const int64_t *__restrict__ key_off, uint32_t R,
             uint64_t key_capacity, uint32_t *__restrict__ slots, int32_t *__restrict__ hit, int32_t *status) {
    pk::pdl_launch_dependents();
    pk::pdl_wait();
    const uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t lane = threadIdx.x & 31;
    if (r >= R) return;  // uniform per warp
    const int64_t a = __ldg(key_off + r);
    int64_t b = __ldg(key_off + r + 1);
    if ((uint64_t)b > key_capacity) b = (int64_t)key_capacity;
    int64_t h = -1;
    bool limit = false;
    for (int64_t base = a; base < b; base += 32) {
        const int64_t g = base + lane;
        uint32_t slot = PK_NO_SLOT;
        if (g < b) {
            const uint4 key = __ldg(reinterpret_cast<const uint4 *>(keys + 32 * g));
            if (!probe(table, mask, max_probe, key, slot)) limit = true;
            slots[g] = slot;
        }
        const uint32_t ball = __ballot_sync(0xffffffffu, g < b && slot == PK_NO_SLOT);
        if (h < 0 && ball) h = base - a + (__ffs(ball) - 1);
    }
    if (h < 0) h = b > a ? b - a : 0;
    if (lane == 0) hit[r] = (int32_t)h;
    if (limit) set_status(status, PK_ERR_PROBE_LIMIT);
}

// One thread per key (few long requests): slots only; k_first_miss follows.
__global__ void __launch_bounds__(256)
k_lookup(const pk_entry *__restrict__ table, uint64_t mask, uint32_t max_probe,
         const uint8_t *__restrict__ keys, const int64_t *__restrict__ key_off, uint32_t R,
         uint64_t key_capacity, uint32_t *__restrict__ slots, int32_t *status) {
    pk::pdl_launch_dependents();
    pk::pdl_wait();
    const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (R == 0 || (uint64_t)g >= key_capacity || g >= __ldg(key_off + R)) return;
    const uint4 key = __ldg(reinterpret_cast<const uint4 *>(keys + 32 * g));
    uint32_t slot;
    if (!probe(table, mask, max_probe, key, slot)) set_status(status, PK_ERR_PROBE_LIMIT);
    slots[g] = slot;
}

// One warp per request: h_r = index of the first PK_NO_SLOT among its keys.
__global__ void __launch_bounds__(256)
k_first_miss(const int64_t *__restrict__ key_off, uint32_t R, uint64_t key_capacity,
             const uint32_t *__restrict__ slots, int32_t *__restrict__ hit) {
    pk::pdl_launch_dependents();
    pk::pdl_wait();
    const uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t lane = threadIdx.x & 31;
    if (r >= R) return;
    const int64_t a = __ldg(key_off + r);
    int64_t b = __ldg(key_off + r + 1);
    if ((uint64_t)b > key_capacity) b = (int64_t)key_capacity;
    int64_t h = b > a ? b - a : 0;
    for (int64_t base = a; base < b; base += 32) {
        const int64_t idx = base + lane;
        const bool miss = idx < b && __ldg(slots + idx) == PK_NO_SLOT;
        const uint32_t ball = __ballot_sync(0xffffffffu, miss);
        if (ball) {
            h = base - a + (__ffs(ball) - 1);
            break;
        }
    }
    if (lane == 0) hit[r] = (int32_t)h;
}

// ---------------------------------------------------------------------------
// Store, kernel 1 of 2: find or claim each key's entry.
//   pre-existing key (epoch of an earlier call): PRESENT with its slot, final
//   key absent: CAS the key into the first empty entry
//   key claimed in this call (by anyone): record the lowest claimant index in
//   `owner` (atomicMax of ~index) and leave PENDING with the entry position
//   in slot_out for kernel 2.
// Capacity: when the table holds few enough entries that this call cannot
// fill it (count + n < capacity), claims are counted once per warp at the
// end.  Otherwise a new key is refused (TABLE_FULL) once the count reaches
// capacity - 1 and every claim is counted as it happens; claims racing at
// that threshold can still take the last empty entries, after which probes
// for absent keys end at max_probe (PK_ERR_PROBE_LIMIT).
// ---------------------------------------------------------------------------
enum Examine { kAdvance, kDone, kClaimedHere };

// Examine entry `ent` (position pos) whose key was read as `cur`.
__device__ __forceinline__ Examine examine(pk_entry *ent, uint64_t pos, uint4 cur, const uint4 &key, uint32_t me,
                                           unsigned long long epoch, bool fast, unsigned long long *counter,
                                           uint64_t capacity, int32_t &res, uint32_t &out) {
    uint4 *kp = reinterpret_cast<uint4 *>(ent->k);
#pragma unroll 1
    for (int pass = 0; pass < 2; ++pass) {
        // A vector load racing a concurrent 128-bit CAS may observe a mix of
        // zero and new words.  When every word is zero or equal to ours, take
        // an atomic snapshot: a CAS that swaps our key for itself changes
        // nothing and returns the entry's whole current key.
        if (!same(cur, key) && !is_zero(cur) && (cur.x == 0 || cur.x == key.x) && (cur.y == 0 || cur.y == key.y) &&
            (cur.z == 0 || cur.z == key.z) && (cur.w == 0 || cur.w == key.w))
            cur = atomicCAS(kp, key, key);
        if (same(cur, key)) {
            const unsigned long long ep = ld_volatile_u64(&ent->epoch);
            if (ep != 0ull && ep != epoch) {  // inserted by an earlier call
                res = PK_STORE_PRESENT;
                out = *(volatile uint32_t *)&ent->slot;
            } else {  // claimed during this call
                atomicMax(&ent->owner, me);
                res = PK_STORE_PENDING;
                out = (uint32_t)pos;
            }
            return kDone;
        }
        if (!is_zero(cur)) return kAdvance;  // a different key holds this entry
        // Room check: refuse a new key once the table holds capacity - 1
        // entries.  Only successful claims are counted (below), so racing
        // duplicates of one key never touch the counter.
        if (!fast && ld_volatile_u64(counter) + 1ull >= capacity) {
            res = PK_ERR_TABLE_FULL;
            return kDone;
        }
        const uint4 old = atomicCAS(kp, make_uint4(0, 0, 0, 0), key);
        if (is_zero(old)) {  // claimed
            *(volatile unsigned long long *)&ent->epoch = epoch;
            atomicMax(&ent->owner, me);
            res = PK_STORE_PENDING;
            out = (uint32_t)pos;
            if (fast) return kClaimedHere;  // counted once per warp at the end
            atomicAdd(counter, 1ull);
            return kDone;
        }
        cur = old;  // examine the winner's key
    }
    return kAdvance;
}

// Insert-if-absent of one entry (index e): result code, output slot/position,
// and whether it claimed an entry that the caller must count (fast mode).
__device__ __forceinline__ void claim(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
                                      unsigned long long *counter, unsigned long long epoch, bool fast,
                                      const uint4 &key, uint32_t my_slot, uint64_t e, int32_t &res, uint32_t &out,
                                      bool &claimed_fast) {
    out = PK_NO_SLOT;
    claimed_fast = false;
    if (is_zero(key)) {
        res = PK_ERR_RESERVED_KEY;
        return;
    }
    if (my_slot == PK_NO_SLOT) {
        res = PK_ERR_ARG;
        return;
    }
    const uint32_t me = ~(uint32_t)e;
    const uint32_t win = mask + 1 < kWin ? (uint32_t)(mask + 1) : kWin;
    const uint64_t pos = home_of(key) & mask;
    uint64_t base = pos & ~(uint64_t)(win - 1);
    uint32_t j0 = (uint32_t)(pos - base);
    uint32_t probed = 0;
    bool done = false;
    res = PK_ERR_PROBE_LIMIT;
    while (!done && probed < max_probe) {
        pk_entry *grp = table + base;
        uint4 v[kWin];
#pragma unroll
        for (uint32_t u = 0; u < kWin; ++u)
            if (u < win) v[u] = ld_volatile_v4(grp[u].k);
#pragma unroll
        for (uint32_t u = 0; u < kWin; ++u) {
            if (u < win && u >= j0 && !done && probed < max_probe) {
                ++probed;
                const Examine x = examine(grp + u, base + u, v[u], key, me, epoch, fast, counter, capacity, res, out);
                if (x != kAdvance) done = true;
                if (x == kClaimedHere) claimed_fast = true;
            }
        }
        base = (base + win) & mask;
        j0 = 0;
    }
}

// List mode, or range mode for few long requests: one thread per entry.
__global__ void __launch_bounds__(256)
k_store_claim(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
              unsigned long long *counter, unsigned long long epoch, const uint8_t *__restrict__ keys,
              const uint32_t *__restrict__ slots, uint64_t n, const int64_t *__restrict__ key_off,
              const int32_t *__restrict__ hit, uint32_t R, int32_t *__restrict__ result,
              uint32_t *__restrict__ slot_out, int32_t *status) {
    // Claims are counted once per block: same-address atomics serialise in L2.
    __shared__ unsigned long long block_claims;
    if (threadIdx.x == 0) block_claims = 0;
    __syncthreads();
    pk::pdl_launch_dependents();
    pk::pdl_wait();
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const uint32_t lane = threadIdx.x & 31;
    const uint64_t e0 = e - lane;
    bool active = e < n;
    if (key_off) {  // range mode: only [key_off[r] + hit[r], key_off[r+1])
        const int64_t total = R > 0 ? __ldg(key_off + R) : 0;
        bool in_range = false;
        if (e0 < n && (int64_t)e0 < total) {
            const uint32_t r = pk::lane_request(key_off, R, (int64_t)e0, total, (int64_t)e);
            if ((int64_t)e < total) {
                const int64_t h = __ldg(hit + r);
                in_range = (int64_t)e - __ldg(key_off + r) >= (h > 0 ? h : 0);
            }
        }
        active = active && in_range;
    }
    unsigned long long cnt = 0;
    if (lane == 0) cnt = ld_volatile_u64(counter);
    const bool fast = __shfl_sync(0xffffffffu, cnt, 0) + n < capacity;
    int32_t res = PK_STORE_SKIPPED;
    uint32_t out = PK_NO_SLOT;
    bool claimed_fast = false;
    if (active) {
        const uint4 key = __ldg(reinterpret_cast<const uint4 *>(keys + 32 * e));
        claim(table, mask, max_probe, capacity, counter, epoch, fast, key, slots[e], e, res, out, claimed_fast);
    }
    if (e < n) {
        result[e] = res;
        slot_out[e] = out;
        if (res < 0) set_status(status, res);
    }
    const uint32_t m = __ballot_sync(0xffffffffu, claimed_fast);
    if (lane == 0 && m) atomicAdd_block(&block_claims, (unsigned long long)__popc(m));
    __syncthreads();
    if (threadIdx.x == 0 && block_claims) atomicAdd(counter, block_claims);
}

// Range mode for many short requests: one warp per request, no search.
// Writes every entry of [key_off[r], key_off[r+1]); entries past key_off[R]
// are marked by the finalize kernel.
__global__ void __launch_bounds__(256)
k_store_claim_req(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
                  unsigned long long *counter, unsigned long long epoch, const uint8_t *__restrict__ keys,
                  const uint32_t *__restrict__ slots, uint64_t n, const int64_t *__restrict__ key_off,
                  const int32_t *__restrict__ hit, uint32_t R, int32_t *__restrict__ result,
                  uint32_t *__restrict__ slot_out, int32_t *status) {
    __shared__ unsigned long long block_claims;  // counted once per block (see k_store_claim)
    if (threadIdx.x == 0) block_claims = 0;
    __syncthreads();
    pk::pdl_launch_dependents();
    pk::pdl_wait();
    const uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t lane = threadIdx.x & 31;
    int64_t a = 0, b = 0, first = 0;
    if (r < R) {  // uniform per warp
        a = __ldg(key_off + r);
        b = __ldg(key_off + r + 1);
        if ((uint64_t)b > n) b = (int64_t)n;
        const int64_t h0 = __ldg(hit + r);
        first = a + (h0 > 0 ? h0 : 0);
    }
    unsigned long long cnt = 0;
    if (lane == 0) cnt = ld_volatile_u64(counter);
    const bool fast = __shfl_sync(0xffffffffu, cnt, 0) + n < capacity;
    uint32_t claimed = 0;
    for (int64_t base = a; base < b; base += 32) {
        const int64_t e = base + lane;
        int32_t res = PK_STORE_SKIPPED;
        uint32_t out = PK_NO_SLOT;
        bool claimed_fast = false;
        if (e < b && e >= first) {
            const uint4 key = __ldg(reinterpret_cast<const uint4 *>(keys + 32 * e));
            claim(table, mask, max_probe, capacity, counter, epoch, fast, key, slots[e], (uint64_t)e, res, out,
                  claimed_fast);
        }
        if (e < b) {
            result[e] = res;
            slot_out[e] = out;
            if (res < 0) set_status(status, res);
        }
        claimed += __popc(__ballot_sync(0xffffffffu, claimed_fast));
    }
    if (lane == 0 && claimed) atomicAdd_block(&block_claims, (unsigned long long)claimed);
    __syncthreads();
    if (threadIdx.x == 0 && block_claims) atomicAdd(counter, block_claims);
}

// Store, kernel 2 of 2: the lowest claimant of each new key writes its slot.
// In range mode, entries past key_off[R] (not keys of this batch) are skipped.
__global__ void __launch_bounds__(256)
k_store_finalize(pk_entry *table, const uint32_t *__restrict__ slots, uint64_t n,
                 const int64_t *__restrict__ key_off, uint32_t R, int32_t *__restrict__ result,
                 uint32_t *__restrict__ slot_out) {
    pk::pdl_launch_dependents();
    pk::pdl_wait();
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= n) return;
    if (key_off && (int64_t)e >= (R > 0 ? __ldg(key_off + R) : 0)) {
        result[e] = PK_STORE_SKIPPED;
        slot_out[e] = PK_NO_SLOT;
        return;
    }
    if (result[e] != PK_STORE_PENDING) return;
    pk_entry *ent = table + slot_out[e];
    const uint32_t winner = ~ent->owner;
    if (winner == (uint32_t)e) {
        ent->slot = slots[e];
        result[e] = PK_STORE_INSERTED;
        slot_out[e] = slots[e];
    } else {
        result[e] = PK_STORE_PRESENT;
        slot_out[e] = slots[winner];
    }
}

// After a table load: every stored entry counts as inserted before any later
// store call (epoch 1; calls on this context use epochs >= 2 from then on).
__global__ void k_mark_loaded(pk_entry *table, uint64_t capacity) {
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < capacity;
         i += (uint64_t)gridDim.x * blockDim.x) {
        const uint4 k = *reinterpret_cast<const uint4 *>(table[i].k);
        table[i].epoch = is_zero(k) ? 0ull : 1ull;
        table[i].owner = 0u;
    }
}

// ---------------------------------------------------------------------------
// Allocation-free store (pk_store_noalloc).  Same insert-if-absent as the
// store above, for callers that own no libpk context: everything a context
// would hold on the device (entry count, call number) and the per-entry claim
// positions live in this one file-scope array, shared by every call.
// ---------------------------------------------------------------------------
struct NoallocScratch {
    unsigned long long count;      // entries in the table (set by the scan, then claims)
    unsigned long long epoch_max;  // largest call number found in the table
    uint32_t pos[PK_NOALLOC_MAX_ENTRIES];  // table position of each PENDING entry
};
static __device__ __align__(256) NoallocScratch g_noalloc_scratch;

// Count the occupied entries and find the latest call number in the table.
__global__ void __launch_bounds__(256)
k_noalloc_scan(const pk_entry *__restrict__ table, uint64_t capacity, NoallocScratch *sc) {
    __shared__ unsigned long long blk_count, blk_epoch;
    if (threadIdx.x == 0) blk_count = blk_epoch = 0;
    __syncthreads();
    unsigned long long cnt = 0, ep = 0;
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < capacity;
         i += (uint64_t)gridDim.x * blockDim.x) {
        const uint4 k = __ldg(reinterpret_cast<const uint4 *>(table[i].k));
        if (!is_zero(k)) {
            ++cnt;
            const unsigned long long e = __ldg(&table[i].epoch);
            ep = e > ep ? e : ep;
        }
    }
    atomicAdd_block(&blk_count, cnt);
    atomicMax_block(&blk_epoch, ep);
    __syncthreads();
    if (threadIdx.x == 0) {
        if (blk_count) atomicAdd(&sc->count, blk_count);
        atomicMax(&sc->epoch_max, blk_epoch);
    }
}

// One thread per entry (list or range mode), as k_store_claim; the call
// number is one past the table's latest and PENDING positions go to scratch.
__global__ void __launch_bounds__(256)
k_noalloc_claim(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity, NoallocScratch *sc,
                const uint8_t *__restrict__ keys, const uint32_t *__restrict__ slots, uint64_t n,
                const int64_t *__restrict__ key_off, const int32_t *__restrict__ hit, uint32_t R,
                int32_t *__restrict__ result, uint32_t *__restrict__ slot_out, int32_t *status) {
    __shared__ unsigned long long block_claims;
    if (threadIdx.x == 0) block_claims = 0;
    __syncthreads();
    const unsigned long long epoch = ld_volatile_u64(&sc->epoch_max) + 1ull;
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const uint32_t lane = threadIdx.x & 31;
    const uint64_t e0 = e - lane;
    bool active = e < n;
    if (key_off) {
        const int64_t total = R > 0 ? __ldg(key_off + R) : 0;
        bool in_range = false;
        if (e0 < n && (int64_t)e0 < total) {
            const uint32_t r = pk::lane_request(key_off, R, (int64_t)e0, total, (int64_t)e);
            if ((int64_t)e < total) {
                const int64_t h = __ldg(hit + r);
                in_range = (int64_t)e - __ldg(key_off + r) >= (h > 0 ? h : 0);
            }
        }
        active = active && in_range;
    }
    unsigned long long cnt = 0;
    if (lane == 0) cnt = ld_volatile_u64(&sc->count);
    const bool fast = __shfl_sync(0xffffffffu, cnt, 0) + n < capacity;
    int32_t res = PK_STORE_SKIPPED;
    uint32_t out = PK_NO_SLOT;
    bool claimed_fast = false;
    if (active) {
        const uint4 key = __ldg(reinterpret_cast<const uint4 *>(keys + 32 * e));
        claim(table, mask, max_probe, capacity, &sc->count, epoch, fast, key, slots[e], e, res, out, claimed_fast);
    }
    if (e < n) {
        result[e] = res;
        if (res == PK_STORE_PENDING) {
            sc->pos[e] = out;
            slot_out[e] = PK_NO_SLOT;
        } else {
            slot_out[e] = out;
        }
        if (res < 0) set_status(status, res);
    }
    const uint32_t m = __ballot_sync(0xffffffffu, claimed_fast);
    if (lane == 0 && m) atomicAdd_block(&block_claims, (unsigned long long)__popc(m));
    __syncthreads();
    if (threadIdx.x == 0 && block_claims) atomicAdd(&sc->count, block_claims);
}

__global__ void __launch_bounds__(256)
k_noalloc_finalize(pk_entry *table, const NoallocScratch *sc, const uint32_t *__restrict__ slots, uint64_t n,
                   int32_t *__restrict__ result, uint32_t *__restrict__ slot_out) {
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= n || result[e] != PK_STORE_PENDING) return;
    pk_entry *ent = table + sc->pos[e];
    const uint32_t winner = ~ent->owner;
    if (winner == (uint32_t)e) {
        ent->slot = slots[e];
        result[e] = PK_STORE_INSERTED;
        slot_out[e] = slots[e];
    } else {
        result[e] = PK_STORE_PRESENT;
        slot_out[e] = slots[winner];
    }
}

unsigned grid_for(uint64_t n, unsigned block) { return (unsigned)((n + block - 1) / block); }

// Per-request kernels when the batch has many short requests; per-key kernels
// when a few requests carry many keys each (a warp per request would then
// walk them serially).
bool per_request(uint32_t R, uint64_t key_capacity) { return R >= 1024 || key_capacity <= 64ull * R; }

}  // namespace

cudaError_t pk_launch_mark_loaded(const pk_ctx *ctx, cudaStream_t s) {
    const uint64_t blocks = (ctx->capacity + 255) / 256;
    k_mark_loaded<<<(unsigned)(blocks < 152 * 16 ? blocks : 152 * 16), 256, 0, s>>>(ctx->table, ctx->capacity);
    return cudaGetLastError();
}

cudaError_t pk_launch_lookup(const pk_ctx *ctx, const uint8_t *keys, const int64_t *key_off, uint32_t R,
                             uint64_t key_capacity, int32_t *hit_chunks, uint32_t *slots, int32_t *status,
                             cudaStream_t s) {
    if (R == 0) return cudaSuccess;
    const uint64_t mask = ctx->capacity - 1;
    cudaError_t e;
    if (per_request(R, key_capacity)) {
        e = pk_launch(k_lookup_req, grid_for(32ull * R, 256), 256, s, (const pk_entry *)ctx->table, mask,
                      ctx->max_probe, keys, key_off, R, key_capacity, slots, hit_chunks, status);
    } else {
        e = key_capacity == 0 ? cudaSuccess
                              : pk_launch(k_lookup, grid_for(key_capacity, 256), 256, s, (const pk_entry *)ctx->table,
                                          mask, ctx->max_probe, keys, key_off, R, key_capacity, slots, status);
        if (e == cudaSuccess)
            e = pk_launch(k_first_miss, grid_for(32ull * R, 256), 256, s, key_off, R, key_capacity,
                          (const uint32_t *)slots, hit_chunks);
    }
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t pk_launch_store(const pk_ctx *ctx, unsigned long long epoch, const uint8_t *keys,
                            const uint32_t *slots, uint64_t n, const int64_t *key_off,
                            const int32_t *hit_chunks, uint32_t R, int32_t *result, uint32_t *slot_out,
                            int32_t *status, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const uint64_t mask = ctx->capacity - 1;
    cudaError_t e;
    if (key_off && R > 0 && per_request(R, n)) {
        e = pk_launch(k_store_claim_req, grid_for(32ull * R, 256), 256, s, ctx->table, mask, ctx->max_probe,
                      ctx->capacity, ctx->counter_dev, epoch, keys, slots, n, key_off, hit_chunks, R, result,
                      slot_out, status);
    } else {
        e = pk_launch(k_store_claim, grid_for(n, 256), 256, s, ctx->table, mask, ctx->max_probe, ctx->capacity,
                      ctx->counter_dev, epoch, keys, slots, n, key_off, hit_chunks, R, result, slot_out, status);
    }
    if (e == cudaSuccess)
        e = pk_launch(k_store_finalize, grid_for(n, 256), 256, s, ctx->table, slots, n, key_off, R, result, slot_out);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// Device address of the allocation-free store's scratch array, resolved once
// per device (host code cannot use the symbol's host-side name as an address).
static void *noalloc_scratch_addr(int device) {
    static std::mutex mu;
    static void *addr[256] = {};
    if (device < 0 || device >= 256) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[device]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
        addr[device] = p;
    }
    return addr[device];
}

cudaError_t pk_launch_store_noalloc(pk_entry *table, uint32_t capacity_log2, uint32_t max_probe,
                                    const uint8_t *keys, const uint32_t *slots, uint64_t n, const int64_t *key_off,
                                    const int32_t *hit_chunks, uint32_t R, int32_t *result, uint32_t *slot_out,
                                    int32_t *status, cudaStream_t s) {
    int device = -1;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return e;
    NoallocScratch *sc = static_cast<NoallocScratch *>(noalloc_scratch_addr(device));
    if (!sc) return cudaErrorInvalidSymbol;
    if (n == 0) return cudaSuccess;
    const uint64_t capacity = 1ull << capacity_log2;
    // count and epoch_max must start at zero; pos needs no clearing
    e = cudaMemsetAsync(sc, 0, 2 * sizeof(unsigned long long), s);
    if (e != cudaSuccess) return e;
    const uint64_t scan_blocks = (capacity + 255) / 256;
    k_noalloc_scan<<<(unsigned)(scan_blocks < 152 * 8 ? scan_blocks : 152 * 8), 256, 0, s>>>(table, capacity, sc);
    k_noalloc_claim<<<grid_for(n, 256), 256, 0, s>>>(table, capacity - 1, max_probe, capacity, sc, keys, slots, n,
                                                      key_off, hit_chunks, key_off ? R : 0, result, slot_out, status);
    k_noalloc_finalize<<<grid_for(n, 256), 256, 0, s>>>(table, sc, slots, n, result, slot_out);
    return cudaGetLastError();
}
