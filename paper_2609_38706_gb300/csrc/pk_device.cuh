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
