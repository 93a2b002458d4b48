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
// One cooperative launch, one CTA per SM slot, in phases separated by
// bounded grid barriers:
//   1. every CTA reads the entry count and returns at once when it is within
//      the budget (the common step costs one short launch);
//   2. gather: one bit per entry (occupied) and the stamps of occupied
//      entries, compacted into scratch;
//   3. radix select of v over the gathered stamps, 8 passes of 8 bits, most
//      significant first; each pass is a privatised shared-memory histogram
//      of the candidates, and every CTA then picks the same bucket;
//   4. compaction in place, one thread per cluster (maximal run of occupied
//      entries, from the bitmap of phase 2): in probe order, an evicted
//      entry is cleared and its slot reported; a kept entry moves to the
//      first empty position between its home and its own, so that every
//      kept key stays reachable by linear probing.  Clusters are disjoint,
//      so no two threads touch the same entry.
#include <cuda_runtime.h>

#include "pk_device.cuh"
#include "pk_internal.h"

namespace {

constexpr uint32_t kEvThreads = 512;
constexpr uint32_t kSpinLimit = 1u << 23;  // x ~100 ns: a barrier gives up after about a second

struct EvictHeader {  // zeroed by the host before every launch
    unsigned int arrive;
    unsigned int gen;
    unsigned long long n;          // stamps gathered
    unsigned long long n_evicted;  // entries removed
    unsigned long long pad;
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

// Grid-wide barrier with a bounded wait.  Returns false (in every thread of
// the CTA) when the wait gave up; the status word then holds PK_ERR_TIMEOUT.
__device__ bool grid_sync(EvictHeader *h, int32_t *status) {
    __shared__ int ok;
    __syncthreads();
    if (threadIdx.x == 0) {
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
                if (++it > kSpinLimit) {
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

__device__ __forceinline__ bool bit(const uint32_t *bm, uint64_t i) { return (__ldcg(bm + (i >> 5)) >> (i & 31)) & 1u; }

__global__ void __launch_bounds__(kEvThreads)
k_evict(pk_entry *table, unsigned long long *stamps, uint64_t capacity, unsigned long long *counter, uint64_t budget,
        uint64_t keep, EvictHeader *h, uint32_t *bitmap, unsigned long long *list, uint32_t *evicted,
        uint64_t evicted_cap, unsigned long long *n_evicted_out, int32_t *status) {
    __shared__ unsigned int sh_hist[256];
    __shared__ unsigned long long sh_sel[2];
    __shared__ unsigned long long sh_evicted;
    const uint32_t tid = threadIdx.x, lane = tid & 31;
    const uint64_t gtid = (uint64_t)blockIdx.x * blockDim.x + tid;
    const uint64_t nthreads = (uint64_t)gridDim.x * blockDim.x;
    const uint64_t mask = capacity - 1;

    // 1. within the budget: nothing to do
    const unsigned long long count = __ldcg(counter);
    if (count <= budget) {
        if (gtid == 0 && n_evicted_out) *n_evicted_out = 0;
        return;
    }
    if (tid == 0) sh_evicted = 0;

    // 2. gather: occupancy bitmap and the stamps of occupied entries
    const uint64_t nwarps = nthreads / 32;
    for (uint64_t base = (gtid / 32) * 32; base < capacity; base += nwarps * 32) {
        const uint64_t i = base + lane;
        const bool occ = i < capacity && !is_zero(__ldcg(reinterpret_cast<const uint4 *>(table[i].k)));
        const uint32_t word = __ballot_sync(0xffffffffu, occ);
        if (lane == 0) bitmap[base >> 5] = word;
        unsigned long long at = 0;
        if (lane == 0 && word) at = atomicAdd(&h->n, (unsigned long long)__popc(word));
        at = __shfl_sync(0xffffffffu, at, 0);
        if (occ) list[at + __popc(word & ((1u << lane) - 1u))] = __ldcg(stamps + i);
    }
    if (!grid_sync(h, status)) return;
    const unsigned long long n = __ldcg(&h->n);

    if (n > keep) {
        // 3. v = the stamp of ascending rank n - keep - 1
        unsigned long long prefix = 0, rank = n - keep - 1;
        for (int d = 0; d < 8; ++d) {
            const int shift = 56 - 8 * d;
            for (uint32_t b = tid; b < 256; b += blockDim.x) sh_hist[b] = 0;
            __syncthreads();
            for (uint64_t j = gtid; j < n; j += nthreads) {
                const unsigned long long x = __ldcg(list + j);
                if (d == 0 || (x >> (shift + 8)) == prefix) atomicAdd(&sh_hist[(x >> shift) & 255u], 1u);
            }
            __syncthreads();
            for (uint32_t b = tid; b < 256; b += blockDim.x)
                if (sh_hist[b]) atomicAdd(&h->hist[d][b], sh_hist[b]);
            if (!grid_sync(h, status)) return;
            if (tid < 32) {  // bucket holding `rank`: 8 buckets per lane, then a warp scan
                unsigned long long c[8], sum = 0;
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    c[u] = __ldcg(&h->hist[d][lane * 8 + u]);
                    sum += c[u];
                }
                unsigned long long incl = sum;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned long long y = __shfl_up_sync(0xffffffffu, incl, o);
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

        // 4. compaction, one thread per cluster start
        unsigned long long mine = 0;
        for (uint64_t i = gtid; i < capacity; i += nthreads) {
            if (!bit(bitmap, i) || bit(bitmap, (i - 1) & mask)) continue;
            for (uint64_t step = 0; step < capacity; ++step) {
                const uint64_t pos = (i + step) & mask;
                if (!bit(bitmap, pos)) break;  // empty before the call: the cluster ends
                uint4 *ep = reinterpret_cast<uint4 *>(&table[pos]);
                const uint4 k = __ldcg(ep), meta = __ldcg(ep + 1);
                const unsigned long long sp = __ldcg(stamps + pos);
                if (sp <= v) {
                    const unsigned long long at = atomicAdd(&h->n_evicted, 1ull);
                    if (evicted && at < evicted_cap) evicted[at] = meta.x;  // the entry's slot
                    else if (evicted) pk::set_status(status, PK_ERR_ARG);
                    __stcg(ep, make_uint4(0, 0, 0, 0));
                    __stcg(ep + 1, make_uint4(0, 0, 0, 0));
                    __stcg(stamps + pos, 0ull);
                    ++mine;
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
        if (mine) atomicAdd_block(&sh_evicted, mine);
        __syncthreads();
        if (tid == 0 && sh_evicted) atomicAdd(counter, (unsigned long long)(-(long long)sh_evicted));
    }
    if (!grid_sync(h, status)) return;
    if (gtid == 0 && n_evicted_out) *n_evicted_out = __ldcg(&h->n_evicted);
}

}  // namespace

uint64_t pk_evict_scratch_bytes_impl(uint64_t capacity) {
    return kHeaderBytes + bitmap_bytes(capacity) + 8 * capacity;
}

cudaError_t pk_launch_evict(const pk_ctx *ctx, uint64_t budget, uint64_t keep, void *scratch, uint32_t *evicted,
                            uint64_t evicted_cap, unsigned long long *n_evicted, int32_t *status, cudaStream_t s) {
    int dev = 0, sms = 0, per_sm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_evict, kEvThreads, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const unsigned grid = (unsigned)(sms * (per_sm < 2 ? per_sm : 2));  // every CTA resident: the barriers need it
    uint8_t *base = static_cast<uint8_t *>(scratch);
    EvictHeader *h = reinterpret_cast<EvictHeader *>(base);
    uint32_t *bitmap = reinterpret_cast<uint32_t *>(base + kHeaderBytes);
    unsigned long long *list = reinterpret_cast<unsigned long long *>(base + kHeaderBytes + bitmap_bytes(ctx->capacity));
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
    e = cudaLaunchKernelEx(&cfg, k_evict, ctx->table, ctx->stamps, ctx->capacity, ctx->counter_dev, budget, keep, h,
                           bitmap, list, evicted, evicted_cap, n_evicted, status);
    return e != cudaSuccess ? e : cudaGetLastError();
}
