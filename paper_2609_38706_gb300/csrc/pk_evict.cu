// pk_evict.cu -- eviction under a fixed budget (Sec. 6.5, eviction under a
// fixed budget: binding provenance keeps one copy per provenance, so a store
// of fixed size evicts more, and thrashes once the distinct working set
// exceeds it).
//
// Budget mode keeps a last-use stamp per table entry, (epoch << 32) | e:
// the store call's number and the key's index in that call, raised by every
// call that finds or inserts the key (pk_table.cu, examine).  Stamps of
// different entries differ, except the zero stamp of entries never used
// since the stamps were attached.  When the table holds more than `budget`
// entries, pk_evict keeps the entries whose stamp is above v, the (keep+1)-th
// largest stamp, and removes the rest: exactly the least recently used
// entries down to `keep`, the whole group of equal stamps when they tie.
//
// One cooperative launch, every CTA resident, in phases separated by
// bounded grid barriers:
//   1. every CTA reads the entry count and returns at once when it is within
//      the budget (the common step costs one short launch);
//   2. gather: one bit per entry (occupied), and the stamp and slot of every
//      occupied entry compacted into scratch, with the smallest and largest
//      stamp;
//   3. radix select of v over the gathered stamps, 8 bits per pass from the
//      highest byte in which the smallest and largest stamp differ (the bytes
//      above are common to all); each pass is a shared-memory histogram of
//      the candidates with warp-aggregated increments, and every CTA then
//      picks the same bucket;
//   4. the slots of the gathered entries with stamp <= v are compacted into
//      the output (one atomic per warp), and the table is compacted in place,
//      one thread per cluster (maximal run of occupied entries, from the
//      bitmap of phase 2): in probe order, an evicted entry is cleared; a kept
//      entry moves to the first empty position between its home and its own,
//      so that every kept key stays reachable by linear probing.  Clusters
//      are disjoint, so no two threads touch the same entry.
#include <cuda_runtime.h>

#include <mutex>

#include "pk_device.cuh"
#include "pk_internal.h"

namespace {

constexpr uint32_t kEvThreads = 512;
constexpr uint32_t kSpinLimit = 1u << 23;  // x ~100 ns: a barrier gives up after about a second

struct EvictHeader {  // zeroed by the host before every launch
    unsigned int arrive;
    unsigned int gen;
    unsigned long long n;          // entries gathered
    unsigned long long n_evicted;  // entries removed
    unsigned long long inv_min;    // ~(smallest stamp gathered)
    unsigned long long max;        // largest stamp gathered
    unsigned int hist[8][256];
};
constexpr uint64_t kHeaderBytes = (sizeof(EvictHeader) + 255) & ~255ull;

uint64_t bitmap_bytes(uint64_t capacity) { return ((capacity + 31) / 32 * 4 + 255) & ~255ull; }

__device__ __forceinline__ bool is_zero(const uint4 &v) { return (v.x | v.y | v.z | v.w) == 0u; }

__device__ __forceinline__ unsigned int ld_acquire(const unsigned int *p) {
    unsigned int v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// The bound of a launch's barrier waits, and the CTA that withholds its
// arrival at the first barrier (none in a normal launch; the timeout test
// names one, so that the others' waits run out).
struct BarrierBound {
    uint32_t spin_limit;
    uint32_t withheld_cta;
};

// Grid-wide barrier with a bounded wait.  Returns false (in every thread of
// the CTA) when the wait gave up; the status word then holds PK_ERR_TIMEOUT.
// A withheld CTA returns false without arriving.
__device__ bool grid_sync(EvictHeader *h, int32_t *status, const BarrierBound &bb) {
    __shared__ int ok;
    __syncthreads();
    if (threadIdx.x == 0 && blockIdx.x == bb.withheld_cta) ok = 0;
    if (threadIdx.x == 0 && blockIdx.x != bb.withheld_cta) {
        ok = 1;
        const unsigned int g = ld_acquire(&h->gen);
        __threadfence();
        if (atomicAdd(&h->arrive, 1u) == gridDim.x - 1) {
            atomicExch(&h->arrive, 0u);
            __threadfence();
            atomicAdd(&h->gen, 1u);
        } else {
            uint32_t it = 0;
            while (ld_acquire(&h->gen) == g) {
                if (++it > bb.spin_limit) {
                    ok = 0;
                    pk::set_status(status, PK_ERR_TIMEOUT);
                    break;
                }
                __nanosleep(100);
            }
        }
        __threadfence();
    }
    __syncthreads();
    return ok != 0;
}

constexpr uint32_t kPer = 4;  // elements per thread per iteration of the strided loops (loads in flight)

// Block-collective append: thread t contributes c elements; returns the list
// position of its first one, with one atomic on `counter` per CTA.  Every
// thread of the CTA calls it.
__device__ __forceinline__ unsigned long long block_append(uint32_t c, unsigned long long *counter) {
    __shared__ uint32_t sh_warp[kEvThreads / 32];
    __shared__ unsigned long long sh_base;
    const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    uint32_t incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= (uint32_t)o) incl += y;
    }
    if (lane == 31) sh_warp[w] = incl;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t total = 0;
        for (uint32_t u = 0; u < kEvThreads / 32; ++u) {
            const uint32_t x = sh_warp[u];
            sh_warp[u] = total;  // exclusive prefix over warps
            total += x;
        }
        sh_base = total ? atomicAdd(counter, (unsigned long long)total) : 0ull;
    }
    __syncthreads();
    return sh_base + sh_warp[w] + (incl - c);
}

__device__ __forceinline__ bool bit(const uint32_t *bm, uint64_t i) { return (__ldcg(bm + (i >> 5)) >> (i & 31)) & 1u; }

// Bulk prefetch of [p, p + bytes) into L2 (bytes a multiple of 16, p 16-byte aligned).
__device__ __forceinline__ void prefetch_l2(const void *p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// Length of the run of occupied positions (bitmap) starting at s, wrapping
// around the table; at most `capacity`.
__device__ uint64_t run_length(const uint32_t *bitmap, uint64_t s, uint64_t capacity) {
    uint64_t L = 0, p = s;
    while (L < capacity) {
        const uint32_t off = (uint32_t)(p & 31);
        const uint64_t left = min((uint64_t)(32 - off), capacity - p);  // valid bits of this word from p
        const uint32_t wd = __ldcg(bitmap + (p >> 5)) >> off;
        const uint32_t ones = (uint32_t)min((uint64_t)(__ffs(~wd) ? __ffs(~wd) - 1 : 32), left);
        L += ones;
        if (ones < left) break;
        p = (p + ones) & (capacity - 1);
    }
    return L < capacity ? L : capacity;
}

// Compaction of one cluster by one thread, serial form: in probe order an
// evicted entry is cleared, a kept entry moves to the first empty position
// from its home.  Any length; used for clusters longer than kPlanMax.
__device__ __noinline__ void compact_walk(pk_entry *table, unsigned long long *stamps, uint64_t s, uint64_t L, uint64_t mask,
                             unsigned long long v) {
    for (uint64_t step = 0; step < L; ++step) {
        const uint64_t pos = (s + step) & mask;
        uint4 *ep = reinterpret_cast<uint4 *>(&table[pos]);
        const uint4 k = __ldcg(ep), meta = __ldcg(ep + 1);
        const unsigned long long sp = __ldcg(stamps + pos);
        if (sp <= v) {
            __stcg(ep, make_uint4(0, 0, 0, 0));
            __stcg(ep + 1, make_uint4(0, 0, 0, 0));
            __stcg(stamps + pos, 0ull);
            continue;
        }
        const uint64_t home = (((uint64_t)k.y << 32) | k.x) & mask;
        const uint64_t dist = (pos - home) & mask;
        for (uint64_t q = 0; q < dist; ++q) {
            const uint64_t t = (home + q) & mask;
            uint4 *tp = reinterpret_cast<uint4 *>(&table[t]);
            if (is_zero(__ldcg(tp))) {  // first empty position from the home: move there
                __stcg(tp + 1, meta);
                __stcg(tp, k);
                __stcg(stamps + t, sp);
                __stcg(ep, make_uint4(0, 0, 0, 0));
                __stcg(ep + 1, make_uint4(0, 0, 0, 0));
                __stcg(stamps + pos, 0ull);
                break;
            }
        }
    }
}

// Pending moves of one thread, flushed four at a time: the sources' entries
// and stamps are all loaded before any target is stored.  Sources come in
// ascending order and every target lies below its source, so no source is
// overwritten before it is read.
struct MoveRing {
    uint32_t src[4], dst[4];  // positions relative to the cluster start
    uint32_t n = 0;
    __device__ __forceinline__ void flush(pk_entry *table, unsigned long long *stamps, uint64_t s0, uint64_t mask) {
        uint4 kk[4], mm[4];
        unsigned long long ss[4];
#pragma unroll
        for (uint32_t u = 0; u < 4; ++u) {
            if (u < n) {
                const uint64_t pos = (s0 + src[u]) & mask;
                const uint4 *ep = reinterpret_cast<const uint4 *>(&table[pos]);
                kk[u] = __ldcg(ep);
                mm[u] = __ldcg(ep + 1);
                ss[u] = __ldcg(stamps + pos);
            }
        }
#pragma unroll
        for (uint32_t u = 0; u < 4; ++u) {
            if (u < n) {
                const uint64_t t = (s0 + dst[u]) & mask;
                uint4 *tp = reinterpret_cast<uint4 *>(&table[t]);
                __stcg(tp + 1, mm[u]);
                __stcg(tp, kk[u]);
                __stcg(stamps + t, ss[u]);
            }
        }
        n = 0;
    }
};

constexpr uint32_t kPlanMax = 1024;  // longest cluster compact_planned takes

// Compaction of one cluster of L <= kPlanMax entries starting at table
// position s0 (capacity >= 64), planned as in k_evict's window: kept entries in
// probe order take the first free position at or after their home, from the
// evicted bits and distance bytes, 32 positions at a time.  A saturated
// distance (255) is replaced by the exact one, from the entry's key.
__device__ __noinline__ void compact_planned(pk_entry *table, unsigned long long *stamps, const uint32_t *evbm, const uint8_t *dist,
                                uint64_t s0, uint32_t L, uint64_t mask) {
    uint64_t taken[kPlanMax / 64];
    for (uint32_t q = 0; q < kPlanMax / 64; ++q) taken[q] = 0;
    const uint64_t n_words = (mask + 1) / 32;
    MoveRing ring;
    for (uint32_t c = 0; c < L; c += 32) {
        const uint64_t p0 = (s0 + c) & mask;
        const uint32_t off = (uint32_t)(p0 & 31);
        const uint64_t wi = p0 >> 5;
        uint32_t evb = __ldcg(evbm + wi) >> off;
        if (off) evb |= __ldcg(evbm + (wi + 1) % n_words) << (32 - off);
        uint8_t d[32];
#pragma unroll
        for (uint32_t k = 0; k < 32; ++k) d[k] = __ldcg(dist + ((p0 + k) & mask));
        for (uint32_t k = 0; k < 32 && c + k < L; ++k) {
            const uint32_t j = c + k;
            if ((evb >> k) & 1u) continue;
            uint64_t dd = d[k];
            if (dd == 255) {  // saturated: the exact distance from the key (position j is not yet overwritten)
                const uint64_t pos = (s0 + j) & mask;
                const uint4 kj = __ldcg(reinterpret_cast<const uint4 *>(table[pos].k));
                dd = (pos - ((((uint64_t)kj.y << 32) | kj.x) & mask)) & mask;
            }
            const uint32_t hh = dd <= j ? j - (uint32_t)dd : j;
            uint32_t t = j;  // position j itself is free
            for (uint32_t q = hh >> 6; q <= (j >> 6); ++q) {
                uint64_t fr = ~taken[q];
                if (q == (hh >> 6)) fr &= ~0ull << (hh & 63);
                if (fr) {
                    t = q * 64 + __ffsll((long long)fr) - 1;
                    break;
                }
            }
            taken[t >> 6] |= 1ull << (t & 63);
            if (t != j) {
                ring.src[ring.n] = j;
                ring.dst[ring.n] = t;
                if (++ring.n == 4) ring.flush(table, stamps, s0, mask);
            }
        }
    }
    ring.flush(table, stamps, s0, mask);
    for (uint32_t q = 0; q * 64 < L; ++q) {  // positions left empty
        uint64_t z = ~taken[q];
        if (L - q * 64 < 64) z &= (1ull << (L - q * 64)) - 1ull;
        while (z) {
            const uint32_t p = q * 64 + __ffsll((long long)z) - 1;
            z &= z - 1;
            const uint64_t pos = (s0 + p) & mask;
            uint4 *ep = reinterpret_cast<uint4 *>(&table[pos]);
            __stcg(ep, make_uint4(0, 0, 0, 0));
            __stcg(ep + 1, make_uint4(0, 0, 0, 0));
            __stcg(stamps + pos, 0ull);
        }
    }
}

__global__ void __launch_bounds__(kEvThreads, 1)
k_evict(pk_entry *table, unsigned long long *stamps, uint64_t capacity, unsigned long long *counter, uint64_t budget,
        uint64_t keep, EvictHeader *h, uint32_t *bitmap, uint32_t *evbm, uint8_t *dist, unsigned long long *list,
        uint32_t *list_slot, uint32_t *evicted, uint64_t evicted_cap, unsigned long long *n_evicted_out,
        int32_t *status, BarrierBound bb) {
    __shared__ unsigned int sh_hist[256];
    __shared__ unsigned long long sh_sel[2];
    __shared__ unsigned long long sh_removed;
    const uint32_t tid = threadIdx.x, lane = tid & 31;
    const uint64_t gtid = (uint64_t)blockIdx.x * blockDim.x + tid;
    const uint64_t nthreads = (uint64_t)gridDim.x * blockDim.x;
    const uint64_t mask = capacity - 1;
    const uint32_t kFull = 0xffffffffu;
    // CTA-uniform strided loops: iteration `it` covers [it0 + it * span, +kPer*kEvThreads), element
    // u of thread t at offset u*kEvThreads + t (coalesced per u)
    const uint64_t span = nthreads * kPer, it0 = (uint64_t)blockIdx.x * kEvThreads * kPer;

    // 1. within the budget: nothing to do
    const unsigned long long count = __ldcg(counter);
    if (count <= budget) {
        if (gtid == 0 && n_evicted_out) *n_evicted_out = 0;
        return;
    }
    if (tid == 0) sh_removed = 0;

    // 2. gather: occupancy bitmap, stamps and slots of occupied entries, stamp range
    unsigned long long lo = ~0ull, hi = 0;
    if (tid == 0 && it0 < capacity) {
        const uint64_t m = min((uint64_t)kPer * kEvThreads, capacity - it0);
        prefetch_l2(&table[it0], (uint32_t)(m * sizeof(pk_entry)));
        prefetch_l2(stamps + it0, (uint32_t)(m * 8));
    }
    for (uint64_t base = it0; base < capacity; base += span) {
        if (tid == 0 && base + span < capacity) {  // the next iteration's entries and stamps
            const uint64_t m = min((uint64_t)kPer * kEvThreads, capacity - base - span);
            prefetch_l2(&table[base + span], (uint32_t)(m * sizeof(pk_entry)));
            prefetch_l2(stamps + base + span, (uint32_t)(m * 8));
        }
        uint4 k[kPer];
        uint32_t sl[kPer];
        unsigned long long st[kPer];
#pragma unroll
        for (uint32_t u = 0; u < kPer; ++u) {  // every load of the iteration at once (empty entries: stamp 0)
            const uint64_t i = base + u * kEvThreads + tid;
            k[u] = make_uint4(0, 0, 0, 0);
            sl[u] = 0;
            st[u] = 0;
            if (i < capacity) {
                const uint4 *ep = reinterpret_cast<const uint4 *>(&table[i]);
                k[u] = __ldcg(ep);
                sl[u] = __ldcg(&table[i].slot);
                st[u] = __ldcg(stamps + i);
            }
        }
        uint32_t c = 0;
#pragma unroll
        for (uint32_t u = 0; u < kPer; ++u) {
            const uint64_t i = base + u * kEvThreads + tid;
            const bool occ = !is_zero(k[u]);
            const uint32_t word = __ballot_sync(kFull, occ);
            if (lane == 0 && i < capacity) bitmap[i >> 5] = word;
            if (i < capacity) {  // distance from the home position, saturated at 255
                const uint64_t d = (i - ((((uint64_t)k[u].y << 32) | k[u].x) & mask)) & mask;
                dist[i] = occ ? (uint8_t)(d < 255 ? d : 255) : (uint8_t)0;
            }
            c += occ;
        }
        unsigned long long j = block_append(c, &h->n);
#pragma unroll
        for (uint32_t u = 0; u < kPer; ++u) {
            if (!is_zero(k[u])) {
                list[j] = st[u];
                list_slot[j] = sl[u];
                ++j;
                lo = st[u] < lo ? st[u] : lo;
                hi = st[u] > hi ? st[u] : hi;
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long l2 = __shfl_xor_sync(kFull, lo, o), h2 = __shfl_xor_sync(kFull, hi, o);
        lo = l2 < lo ? l2 : lo;
        hi = h2 > hi ? h2 : hi;
    }
    if (lane == 0 && hi >= lo) {
        atomicMax(&h->inv_min, ~lo);
        atomicMax(&h->max, hi);
    }
    if (!grid_sync(h, status, bb)) return;
    const unsigned long long n = __ldcg(&h->n);
    unsigned long long prefix_v = 0;  // v, once selected

    if (n > keep) {
        // 3. v = the stamp of ascending rank n - keep - 1
        const unsigned long long smin = ~__ldcg(&h->inv_min), smax = __ldcg(&h->max);
        const unsigned long long diff = smin ^ smax;
        const int top = diff ? (63 - __clzll((long long)diff)) / 8 : -1;  // highest differing byte
        unsigned long long prefix = top == 7 ? 0ull : top < 0 ? smin : smin >> (8 * (top + 1));
        unsigned long long rank = n - keep - 1;
        for (int byte = top, p = 0; byte >= 0; --byte, ++p) {
            const int shift = 8 * byte;
            for (uint32_t b = tid; b < 256; b += blockDim.x) sh_hist[b] = 0;
            __syncthreads();
            for (uint64_t base = it0; base < n; base += span) {
                unsigned long long x[kPer];
#pragma unroll
                for (uint32_t u = 0; u < kPer; ++u) {
                    const uint64_t j = base + u * kEvThreads + tid;
                    x[u] = j < n ? __ldcg(list + j) : 0ull;
                }
#pragma unroll
                for (uint32_t u = 0; u < kPer; ++u) {
                    const uint64_t j = base + u * kEvThreads + tid;
                    const bool cand = j < n && (byte == top || (x[u] >> (shift + 8)) == prefix);
                    const uint32_t bin = cand ? (uint32_t)(x[u] >> shift) & 255u : 256u;
                    const uint32_t peers = __match_any_sync(kFull, bin);
                    if (bin < 256 && (peers & ((1u << lane) - 1u)) == 0) atomicAdd(&sh_hist[bin], __popc(peers));
                }
            }
            __syncthreads();
            for (uint32_t b = tid; b < 256; b += blockDim.x)
                if (sh_hist[b]) atomicAdd(&h->hist[p][b], sh_hist[b]);
            if (!grid_sync(h, status, bb)) return;
            if (tid < 32) {  // bucket holding `rank`: 8 buckets per lane, then a warp scan
                unsigned long long c[8], sum = 0;
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    c[u] = __ldcg(&h->hist[p][lane * 8 + u]);
                    sum += c[u];
                }
                unsigned long long incl = sum;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned long long y = __shfl_up_sync(kFull, incl, o);
                    if (lane >= (uint32_t)o) incl += y;
                }
                unsigned long long excl = incl - sum;
                if (rank >= excl && rank < incl) {
#pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        if (rank >= excl && rank < excl + c[u]) {
                            sh_sel[0] = lane * 8 + u;
                            sh_sel[1] = rank - excl;
                        }
                        excl += c[u];
                    }
                }
            }
            __syncthreads();
            prefix = (prefix << 8) | sh_sel[0];
            rank = sh_sel[1];
            __syncthreads();
        }
        const unsigned long long v = prefix;
        prefix_v = v;

        // 4a. the slots of the removed entries, one atomic per CTA and iteration
        unsigned long long removed = 0;
        for (uint64_t base = it0; base < n; base += span) {
            bool ev[kPer];
            uint32_t c = 0;
#pragma unroll
            for (uint32_t u = 0; u < kPer; ++u) {
                const uint64_t j = base + u * kEvThreads + tid;
                ev[u] = j < n && __ldcg(list + j) <= v;
                c += ev[u];
            }
            unsigned long long o = block_append(c, &h->n_evicted);
            removed += c;
#pragma unroll
            for (uint32_t u = 0; u < kPer; ++u) {
                if (ev[u]) {
                    const uint64_t j = base + u * kEvThreads + tid;
                    if (o < evicted_cap) evicted[o] = __ldcg(list_slot + j);
                    else if (evicted) pk::set_status(status, PK_ERR_ARG);
                    ++o;
                }
            }
        }
        if (removed) atomicAdd_block(&sh_removed, removed);
        __syncthreads();
        if (tid == 0 && sh_removed) atomicAdd(counter, (unsigned long long)(-(long long)sh_removed));

        // 4b. the evicted positions as a bitmap
        for (uint64_t base = it0; base < capacity; base += span) {
            unsigned long long st[kPer];
            uint32_t wd[kPer];
#pragma unroll
            for (uint32_t u = 0; u < kPer; ++u) {
                const uint64_t i = base + u * kEvThreads + tid;
                st[u] = i < capacity ? __ldcg(stamps + i) : 0ull;
                wd[u] = i < capacity ? __ldcg(bitmap + (i >> 5)) : 0u;
            }
#pragma unroll
            for (uint32_t u = 0; u < kPer; ++u) {
                const uint64_t i = base + u * kEvThreads + tid;
                const bool ev = ((wd[u] >> lane) & 1u) && st[u] <= v;
                const uint32_t word = __ballot_sync(kFull, ev);
                if (lane == 0 && i < capacity) evbm[i >> 5] = word;
            }
        }
    }
    if (!grid_sync(h, status, bb)) return;
    if (n > keep) {
        // 4c. compaction: one thread per bitmap word, for the clusters that start in it.  Clusters
        // that end within the 64 positions of the word and the next one are planned in registers
        // from the occupancy, evicted and distance bytes; the word's moves then go out four loads
        // at a time.  Longer clusters take compact_planned (the same plan, 32 positions at a time),
        // tables below 64 entries and clusters beyond kPlanMax compact_walk.
        const unsigned long long v = prefix_v;
        const uint64_t n_words = (capacity + 31) / 32;
        for (uint64_t w = gtid; w < n_words; w += nthreads) {
            const uint32_t occ_lo = __ldcg(bitmap + w);
            if (!occ_lo) continue;
            const uint32_t before = bit(bitmap, (w * 32 + mask) & mask);  // the position before bit 0
            uint32_t starts = occ_lo & ~((occ_lo << 1) | before);
            if (capacity < 64) {
                while (starts) {
                    const uint32_t b = __ffs(starts) - 1;
                    starts &= starts - 1;
                    compact_walk(table, stamps, w * 32 + b, run_length(bitmap, w * 32 + b, capacity), mask, v);
                }
                continue;
            }
            const uint64_t w1 = (w + 1) % n_words;  // the next word (wrapping)
            const uint64_t occ = occ_lo | ((uint64_t)__ldcg(bitmap + w1) << 32);
            const uint64_t evw = __ldcg(evbm + w) | ((uint64_t)__ldcg(evbm + w1) << 32);
            uint32_t dv[16];
            {
                const uint4 *d0 = reinterpret_cast<const uint4 *>(dist + w * 32);
                const uint4 *d1 = reinterpret_cast<const uint4 *>(dist + w1 * 32);
                const uint4 a0 = __ldcg(d0), a1 = __ldcg(d0 + 1), b0 = __ldcg(d1), b1 = __ldcg(d1 + 1);
                dv[0] = a0.x, dv[1] = a0.y, dv[2] = a0.z, dv[3] = a0.w, dv[4] = a1.x, dv[5] = a1.y, dv[6] = a1.z;
                dv[7] = a1.w, dv[8] = b0.x, dv[9] = b0.y, dv[10] = b0.z, dv[11] = b0.w, dv[12] = b1.x;
                dv[13] = b1.y, dv[14] = b1.z, dv[15] = b1.w;
            }
            // window position p (0..63) is table position (w * 32 + p) & mask
            uint64_t zero = 0, msrc = 0;
            uint8_t dst_of[64];
            while (starts) {
                const uint32_t b = __ffs(starts) - 1;
                starts &= starts - 1;
                const uint64_t rest = ~(occ >> b);
                const uint32_t run = rest ? __ffsll((long long)rest) - 1 : 64 - b;
                if (b + run < 64) {  // the cluster ends inside the window
                    uint64_t taken = 0;  // relative to b
                    for (uint32_t j = 0; j < run; ++j) {
                        const uint32_t p = b + j;
                        if ((evw >> p) & 1u) continue;
                        const uint32_t d = (dv[p >> 2] >> (8 * (p & 3))) & 255u;
                        const uint32_t hh = d <= j ? j - d : j;
                        const uint32_t t = __ffsll((long long)(~taken & (~0ull << hh))) - 1;
                        taken |= 1ull << t;
                        if (t != j) {
                            msrc |= 1ull << p;
                            dst_of[p] = (uint8_t)(b + t);
                        }
                    }
                    zero |= (((1ull << run) - 1ull) & ~taken) << b;
                } else {  // a longer cluster
                    const uint64_t L = run_length(bitmap, w * 32 + b, capacity);
                    if (L <= kPlanMax)
                        compact_planned(table, stamps, evbm, dist, w * 32 + b, (uint32_t)L, mask);
                    else
                        compact_walk(table, stamps, w * 32 + b, L, mask, v);
                }
            }
            // moves in ascending order, four loads before their stores: a target is below its
            // source, so every source is read before anything overwrites it
            while (msrc) {
                uint32_t src[4];
                uint4 kk[4], mm[4];
                unsigned long long ss[4];
                uint32_t cnt = 0;
#pragma unroll
                for (uint32_t u = 0; u < 4; ++u) {
                    if (msrc) {
                        src[u] = __ffsll((long long)msrc) - 1;
                        msrc &= msrc - 1;
                        const uint64_t pos = (w * 32 + src[u]) & mask;
                        const uint4 *ep = reinterpret_cast<const uint4 *>(&table[pos]);
                        kk[u] = __ldcg(ep);
                        mm[u] = __ldcg(ep + 1);
                        ss[u] = __ldcg(stamps + pos);
                        cnt = u + 1;
                    }
                }
#pragma unroll
                for (uint32_t u = 0; u < 4; ++u) {
                    if (u < cnt) {
                        const uint64_t t = (w * 32 + dst_of[src[u]]) & mask;
                        uint4 *tp = reinterpret_cast<uint4 *>(&table[t]);
                        __stcg(tp + 1, mm[u]);
                        __stcg(tp, kk[u]);
                        __stcg(stamps + t, ss[u]);
                    }
                }
            }
            while (zero) {  // positions left empty: evicted, or vacated and not retaken
                const uint32_t p = __ffsll((long long)zero) - 1;
                zero &= zero - 1;
                const uint64_t pos = (w * 32 + p) & mask;
                uint4 *ep = reinterpret_cast<uint4 *>(&table[pos]);
                __stcg(ep, make_uint4(0, 0, 0, 0));
                __stcg(ep + 1, make_uint4(0, 0, 0, 0));
                __stcg(stamps + pos, 0ull);
            }
        }
    }
    if (!grid_sync(h, status, bb)) return;
    if (gtid == 0 && n_evicted_out) *n_evicted_out = __ldcg(&h->n_evicted);
}

}  // namespace

uint64_t pk_evict_scratch_bytes_impl(uint64_t capacity) {
    return kHeaderBytes + 2 * bitmap_bytes(capacity) + 8 * capacity + 4 * capacity + ((capacity + 255) & ~255ull);
}

// Resident CTAs of k_evict on a device (SMs x CTAs per SM), computed once per device.
static cudaError_t evict_resident(int dev, uint64_t *out) {
    static std::mutex mu;
    static uint64_t cache[256] = {};
    if (dev < 0 || dev >= 256) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!cache[dev]) {
        int sms = 0, per_sm = 0;
        cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_evict, kEvThreads, 0);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) return cudaErrorInvalidConfiguration;
        cache[dev] = (uint64_t)sms * per_sm;
    }
    *out = cache[dev];
    return cudaSuccess;
}

cudaError_t pk_launch_evict(const pk_ctx *ctx, uint64_t budget, uint64_t keep, void *scratch, uint32_t *evicted,
                            uint64_t evicted_cap, unsigned long long *n_evicted, int32_t *status, cudaStream_t s,
                            uint32_t spin_limit, bool withhold_first_cta) {
    int dev = 0;
    uint64_t resident = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = evict_resident(dev, &resident);
    if (e != cudaSuccess) return e;
    // every CTA resident (the barriers need it); no more CTAs than the table has rows of kEvThreads entries
    const uint64_t want = (ctx->capacity + kEvThreads - 1) / kEvThreads;
    const unsigned grid = (unsigned)(want < resident ? want : resident);
    uint8_t *base = static_cast<uint8_t *>(scratch);
    EvictHeader *h = reinterpret_cast<EvictHeader *>(base);
    uint32_t *bitmap = reinterpret_cast<uint32_t *>(base + kHeaderBytes);
    const uint64_t bmb = bitmap_bytes(ctx->capacity);
    uint32_t *evbm = reinterpret_cast<uint32_t *>(base + kHeaderBytes + bmb);
    uint8_t *dist = base + kHeaderBytes + 2 * bmb;
    unsigned long long *list =
        reinterpret_cast<unsigned long long *>(dist + ((ctx->capacity + 255) & ~255ull));
    uint32_t *list_slot = reinterpret_cast<uint32_t *>(list + ctx->capacity);
    e = cudaMemsetAsync(h, 0, sizeof(EvictHeader), s);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kEvThreads);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const BarrierBound bb{spin_limit == 0 || spin_limit > kSpinLimit ? kSpinLimit : spin_limit,
                          withhold_first_cta ? 0u : 0xffffffffu};
    e = cudaLaunchKernelEx(&cfg, k_evict, ctx->table, ctx->stamps, ctx->capacity, ctx->counter_dev, budget, keep, h,
                           bitmap, evbm, dist, list, list_slot, evicted, evicted_cap, n_evicted, status, bb);
    return e != cudaSuccess ? e : cudaGetLastError();
}
