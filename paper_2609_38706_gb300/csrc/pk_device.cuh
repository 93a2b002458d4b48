// pk_device.cuh -- small device helpers shared by the libpk kernels.
#pragma once
#include <stdint.h>

#include "../../include/pk.h"

namespace pk {

__device__ __forceinline__ void set_status(int32_t *status, int32_t code) {
    if (status) atomicCAS(status, 0, code);
}

// Request index r with key_off[r] <= g < key_off[r+1], for a non-decreasing
// key_off with key_off[0] <= g < key_off[R].  Called by all 32 lanes of a warp
// with the same g: each level probes 32 positions at once, so R = 2^14
// requests resolve in 3 rounds of independent loads instead of 14 dependent
// ones.
__device__ __forceinline__ uint32_t warp_find_request(const int64_t *key_off, uint32_t R,
                                                      int64_t g) {
    const uint32_t lane = threadIdx.x & 31;
    uint32_t lo = 0, hi = R;  // key_off[lo] <= g < key_off[hi]
    while (hi - lo > 1) {
        const uint32_t span = hi - lo;
        const uint32_t step = span > 32 ? span / 32 : 1;  // span <= 32: every candidate probed at once
        uint32_t p = lo + (lane + 1) * step;
        if (p > hi - 1) p = hi - 1;
        const bool le = __ldcg(key_off + p) <= g;
        const uint32_t ball = __ballot_sync(0xffffffffu, le);
        // probes are non-decreasing in lane, so the set lanes form a prefix
        const int last = 31 - __clz(ball);  // -1 if none
        const uint32_t new_lo = last >= 0 ? __shfl_sync(0xffffffffu, p, last) : lo;
        const int next = last + 1;
        const uint32_t new_hi = next <= 31 ? __shfl_sync(0xffffffffu, p, next) : hi;
        lo = new_lo;
        hi = (new_hi > lo) ? new_hi : hi;
        if (span <= 32) break;
    }
    return lo;
}

// Same, for one thread, restricted to [lo, hi) known to contain the answer.
__device__ __forceinline__ uint32_t find_request_in(const int64_t *key_off, uint32_t lo, uint32_t hi,
                                                    int64_t g) {
    while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (__ldcg(key_off + mid) <= g) lo = mid; else hi = mid;
    }
    return lo;
}

// Per-lane request of item g (items of one warp are g0 .. g0+31, g0 the
// warp's first item, all lanes active).  `total` = key_off[R].
__device__ __forceinline__ uint32_t lane_request(const int64_t *key_off, uint32_t R, int64_t g0,
                                                 int64_t total, int64_t g) {
    const uint32_t r0 = warp_find_request(key_off, R, g0);
    int64_t g_last = g0 + 31;
    if (g_last >= total) g_last = total - 1;
    const uint32_t r1 = warp_find_request(key_off, R, g_last);
    return find_request_in(key_off, r0, r1 + 1, g < total ? g : total - 1);
}

// Same result as lane_request with one search: r0 (the request of the warp's
// first item) by warp_find_request, then one 32-wide load of key_off[r0+1 ..]
// and a search over those 32 values by shuffles (non-decreasing key_off: r = r0
// + the count of them <= g, one of 33 outcomes: 6 halvings).  A lane whose item
// lies past those 32 requests (only after runs of empty requests) falls back to
// find_request_in.
__device__ __forceinline__ uint32_t lane_request_window(const int64_t *key_off, uint32_t R, int64_t g0,
                                                        int64_t total, int64_t g) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t r0 = warp_find_request(key_off, R, g0);
    const uint64_t p = (uint64_t)r0 + 1 + lane;
    const int64_t v = p <= R ? __ldcg(key_off + p) : INT64_MAX;
    const int64_t gg = g < total ? g : total - 1;
    int lo = 0, hi = 32;  // the first j with key_off[r0 + 1 + j] > gg lies in [lo, hi] (32: none of the 32)
#pragma unroll
    for (int it = 0; it < 6; ++it) {
        const int mid = (lo + hi) >> 1;
        const int64_t vm = __shfl_sync(0xffffffffu, v, mid < 31 ? mid : 31);
        if (lo < hi) {
            if (vm <= gg) lo = mid + 1; else hi = mid;
        }
    }
    if (lo < 32) return r0 + (uint32_t)lo;
    return find_request_in(key_off, r0 + 32, R, gg);
}

// Same result again, for batches of about equal requests: a guess from the mean
// request size, r_g = g0 * R / total, one 32-wide load of key_off[w0 ..] with
// w0 = r_g - 8, and the same shuffle search; used when that window brackets
// every lane's item, else lane_request_window.
__device__ __forceinline__ uint32_t lane_request_guess(const int64_t *key_off, uint32_t R, int64_t g0,
                                                       int64_t total, int64_t g) {
    const uint32_t lane = threadIdx.x & 31;
    const int64_t gg = g < total ? g : total - 1;
    uint32_t rg = (uint32_t)((float)g0 / (float)total * (float)R);
    rg = rg >= R ? R - 1 : rg;
    const uint32_t w0 = rg > 8 ? rg - 8 : 0;
    const uint64_t p = (uint64_t)w0 + lane;
    const int64_t u = p <= R ? __ldcg(key_off + p) : INT64_MAX;
    const int64_t u0 = __shfl_sync(0xffffffffu, u, 0);
    int lo = 1, hi = 32;  // the first j >= 1 with key_off[w0 + j] > gg lies in [lo, hi] (32: none of the 31)
#pragma unroll
    for (int it = 0; it < 6; ++it) {
        const int mid = (lo + hi) >> 1;
        const int64_t vm = __shfl_sync(0xffffffffu, u, mid < 31 ? mid : 31);
        if (lo < hi) {
            if (vm <= gg) lo = mid + 1; else hi = mid;
        }
    }
    if (__all_sync(0xffffffffu, u0 <= g0 && lo < 32)) return w0 + (uint32_t)lo - 1;
    return lane_request_window(key_off, R, g0, total, g);
}

}  // namespace pk

namespace pk {

// Programmatic dependent launch (sm_90+).  Every libpk kernel is launched with
// programmatic stream serialization: it may become resident while the previous
// kernel of the stream drains, and waits for its predecessor's completion (and
// memory) before touching global memory.  Kernels release their successor
// once their main work is done (short kernels at their start): a successor
// released early sits on the SMs, with its own successor, for the whole run of
// the kernel (multi-adapter batch: key derivation 82 -> 74 us, small-block
// step 1073 -> 909 us when the digest and chain kernels release late).  Both
// are no-ops for a kernel launched without the attribute.
//
// Memory written by a predecessor is read only with coherent loads (plain or
// L2 loads: __ldcg, ld.global.cg), never through the non-coherent read-only
// path (__ldg, ld.global.nc, loads through const __restrict__ pointers): a
// kernel resident while its predecessor still writes can read stale data on
// that path even after the wait (measured: a store in range mode reading the
// lookup's h_r as 0).  pdl_wait(p...) also passes the kernel's pointers
// through an empty asm after the wait, so that no access through them is
// scheduled before it.
template <typename P>
__device__ __forceinline__ void launder(P &p) {
    asm volatile("" : "+l"(p));
}
template <typename... P>
__device__ __forceinline__ void pdl_wait(P &...p) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    (launder(p), ...);
}
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

}  // namespace pk
