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

#include "pk_internal.h"

namespace {

__device__ __forceinline__ void set_status(int32_t *status, int32_t code) {
    if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ bool is_zero(const uint4 &v) { return (v.x | v.y | v.z | v.w) == 0u; }
__device__ __forceinline__ bool same(const uint4 &a, const uint4 &b) {
    return ((a.x ^ b.x) | (a.y ^ b.y) | (a.z ^ b.z) | (a.w ^ b.w)) == 0u;
}
__device__ __forceinline__ uint64_t home_of(const uint4 &k) {
    return ((uint64_t)k.y << 32) | k.x;  // bytes 0..7, little-endian
}

__device__ __forceinline__ uint32_t find_request(const int64_t *__restrict__ key_off, uint32_t R,
                                                 int64_t g) {
    uint32_t lo = 0, hi = R;  // key_off[lo] <= g < key_off[hi]
    while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (__ldg(key_off + mid) <= g) lo = mid; else hi = mid;
    }
    return lo;
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

// ---------------------------------------------------------------------------
// Lookup
// ---------------------------------------------------------------------------
__global__ void k_hit_init(const int64_t *__restrict__ key_off, uint32_t R, int32_t *__restrict__ hit) {
    const uint32_t r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r < R) hit[r] = (int32_t)(key_off[r + 1] - key_off[r]);
}

__global__ void __launch_bounds__(256)
k_lookup(const pk_entry *__restrict__ table, uint64_t mask, uint32_t max_probe,
         const uint8_t *__restrict__ keys, const int64_t *__restrict__ key_off, uint32_t R,
         int32_t *hit, uint32_t *__restrict__ slots, int32_t *status) {
    const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (R == 0 || g >= __ldg(key_off + R)) return;
    const uint4 key = __ldg(reinterpret_cast<const uint4 *>(keys + 32 * g));
    uint32_t slot = PK_NO_SLOT;
    if (!is_zero(key)) {
        const uint64_t home = home_of(key);
        uint32_t s = 0;
        for (; s < max_probe; ++s) {
            const pk_entry *e = table + ((home + s) & mask);
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(e->k));
            if (same(v, key)) {
                slot = __ldg(&e->slot);
                break;
            }
            if (is_zero(v)) break;
        }
        if (s == max_probe) set_status(status, PK_ERR_PROBE_LIMIT);
    }
    slots[g] = slot;
    if (slot == PK_NO_SLOT) {
        const uint32_t r = find_request(key_off, R, g);
        atomicMin(hit + r, (int32_t)(g - __ldg(key_off + r)));
    }
}

// ---------------------------------------------------------------------------
// Store, kernel 1 of 2: find or claim each key's entry.
//   pre-existing key (epoch of an earlier call): PRESENT with its slot, final
//   key absent: reserve capacity, CAS the key into the first empty entry
//   key claimed in this call (by anyone): record the lowest claimant index in
//   `owner` (atomicMax of ~index) and leave PENDING with the entry position
//   in slot_out for kernel 2.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
k_store_claim(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
              unsigned long long *counter, unsigned long long epoch, const uint8_t *__restrict__ keys,
              const uint32_t *__restrict__ slots, uint64_t n, const int64_t *__restrict__ key_off,
              const int32_t *__restrict__ hit, uint32_t R, int32_t *__restrict__ result,
              uint32_t *__restrict__ slot_out, int32_t *status) {
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= n) return;
    if (key_off) {  // range mode: only [key_off[r] + hit[r], key_off[r+1])
        bool active = false;
        if (R > 0 && (int64_t)e < __ldg(key_off + R)) {
            const uint32_t r = find_request(key_off, R, (int64_t)e);
            const int64_t h = __ldg(hit + r);
            active = (int64_t)e - __ldg(key_off + r) >= (h > 0 ? h : 0);
        }
        if (!active) {
            result[e] = PK_STORE_SKIPPED;
            slot_out[e] = PK_NO_SLOT;
            return;
        }
    }
    const uint4 key = __ldg(reinterpret_cast<const uint4 *>(keys + 32 * e));
    const uint32_t my_slot = slots[e];
    int32_t res = 0;
    uint32_t out = PK_NO_SLOT;
    if (is_zero(key)) {
        res = PK_ERR_RESERVED_KEY;
    } else if (my_slot == PK_NO_SLOT) {
        res = PK_ERR_ARG;
    } else {
        const uint32_t me = ~(uint32_t)e;
        const uint64_t home = home_of(key);
        res = PK_ERR_PROBE_LIMIT;
        uint32_t s = 0;
        while (s < max_probe) {
            const uint64_t pos = (home + s) & mask;
            pk_entry *ent = table + pos;
            uint4 *kp = reinterpret_cast<uint4 *>(ent->k);
            uint4 v = ld_volatile_v4(ent->k);
            // A vector load racing a concurrent 128-bit CAS may observe a mix of
            // zero and new words.  When every word is zero or equal to ours, take
            // an atomic snapshot instead: a CAS that swaps our key for itself
            // changes nothing and returns the entry's whole current key.
            if (!same(v, key) && !is_zero(v) && (v.x == 0 || v.x == key.x) && (v.y == 0 || v.y == key.y) &&
                (v.z == 0 || v.z == key.z) && (v.w == 0 || v.w == key.w))
                v = atomicCAS(kp, key, key);
            if (same(v, key)) {
                const unsigned long long ep = ld_volatile_u64(&ent->epoch);
                if (ep != 0ull && ep != epoch) {  // inserted by an earlier call
                    res = PK_STORE_PRESENT;
                    out = *(volatile uint32_t *)&ent->slot;
                } else {  // claimed during this call
                    atomicMax(&ent->owner, me);
                    res = PK_STORE_PENDING;
                    out = (uint32_t)pos;
                }
                break;
            }
            if (is_zero(v)) {
                const unsigned long long c = atomicAdd(counter, 1ull);
                if (c + 1ull >= capacity) {  // would leave no empty entry
                    atomicAdd(counter, ~0ull);
                    res = PK_ERR_TABLE_FULL;
                    break;
                }
                const uint4 old = atomicCAS(kp, make_uint4(0, 0, 0, 0), key);
                if (is_zero(old)) {  // claimed
                    *(volatile unsigned long long *)&ent->epoch = epoch;
                    atomicMax(&ent->owner, me);
                    res = PK_STORE_PENDING;
                    out = (uint32_t)pos;
                    break;
                }
                atomicAdd(counter, ~0ull);  // release the reservation
                if (same(old, key)) {       // another entry of this call claimed it first
                    atomicMax(&ent->owner, me);
                    res = PK_STORE_PENDING;
                    out = (uint32_t)pos;
                    break;
                }
            }
            ++s;  // a different key holds this entry
        }
    }
    result[e] = res;
    slot_out[e] = out;
    if (res < 0) set_status(status, res);
}

// Store, kernel 2 of 2: the lowest claimant of each new key writes its slot.
__global__ void __launch_bounds__(256)
k_store_finalize(pk_entry *table, const uint32_t *__restrict__ slots, uint64_t n,
                 int32_t *__restrict__ result, uint32_t *__restrict__ slot_out) {
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= n || result[e] != PK_STORE_PENDING) return;
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

unsigned grid_for(uint64_t n, unsigned block) { return (unsigned)((n + block - 1) / block); }

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
    k_hit_init<<<grid_for(R, 256), 256, 0, s>>>(key_off, R, hit_chunks);
    if (key_capacity > 0)
        k_lookup<<<grid_for(key_capacity, 256), 256, 0, s>>>(ctx->table, ctx->capacity - 1, ctx->max_probe, keys,
                                                             key_off, R, hit_chunks, slots, status);
    return cudaGetLastError();
}

cudaError_t pk_launch_store(const pk_ctx *ctx, unsigned long long epoch, const uint8_t *keys,
                            const uint32_t *slots, uint64_t n, const int64_t *key_off,
                            const int32_t *hit_chunks, uint32_t R, int32_t *result, uint32_t *slot_out,
                            int32_t *status, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const unsigned grid = grid_for(n, 256);
    k_store_claim<<<grid, 256, 0, s>>>(ctx->table, ctx->capacity - 1, ctx->max_probe, ctx->capacity,
                                       ctx->counter_dev, epoch, keys, slots, n, key_off, hit_chunks, R, result,
                                       slot_out, status);
    k_store_finalize<<<grid, 256, 0, s>>>(ctx->table, slots, n, result, slot_out);
    return cudaGetLastError();
}
