// pk_pages.cu -- store-side differential omission checker (sec. 6.3 of the
// paper; Eq. 4): two workers that differ in one dimension write pages for the
// same documents; a key of one worker that the other also wrote, with page
// bytes that differ, means the key omits a dimension that changes the state.
// The join on keys is a table lookup (pk_table.cu); this file compares the
// joined pages.
#include <cuda_runtime.h>

#include "pk_device.cuh"
#include "pk_internal.h"

namespace {

constexpr int kCmpThreads = 256;
constexpr int kCmpUnroll = 4;  // 16-byte loads in flight per lane and page

// One warp per page pair.  verdict[j] = PK_PAGE_ABSENT when slots[j] is
// PK_NO_SLOT, else PK_PAGE_EQUAL or PK_PAGE_DIFFERS after reading all
// page_bytes of pages[j] and ref_pages[slots[j]] (no early exit: every page
// pair costs the same two page reads).  counts[v] += keys with verdict v.
__global__ void __launch_bounds__(kCmpThreads)
k_compare_pages(const uint32_t *slots, const uint8_t *pages, const uint8_t *ref_pages, uint64_t n, uint64_t n_ref,
                uint64_t page_bytes, int32_t *verdict, unsigned long long *counts, int32_t *status) {
    __shared__ unsigned long long block_counts[3];
    if (threadIdx.x < 3) block_counts[threadIdx.x] = 0;
    __syncthreads();
    pk::pdl_wait(slots, pages, ref_pages, verdict, counts, status);
    const uint64_t j = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t lane = threadIdx.x & 31;
    if (j < n) {  // uniform per warp
        const uint32_t slot = __ldcg(slots + j);
        int32_t v = PK_PAGE_ABSENT;
        if (slot != PK_NO_SLOT && slot >= n_ref) {
            if (lane == 0) pk::set_status(status, PK_ERR_ARG);  // the slot names no reference page
        } else if (slot != PK_NO_SLOT) {
            const uint4 *a = reinterpret_cast<const uint4 *>(pages + j * page_bytes);
            const uint4 *b = reinterpret_cast<const uint4 *>(ref_pages + (uint64_t)slot * page_bytes);
            const uint64_t words = page_bytes / 16;
            uint32_t diff = 0;
            for (uint64_t w0 = lane; w0 < words; w0 += 32 * kCmpUnroll) {
                uint4 x[kCmpUnroll], y[kCmpUnroll];
#pragma unroll
                for (int u = 0; u < kCmpUnroll; ++u) {
                    const uint64_t w = w0 + 32ull * u;
                    x[u] = y[u] = make_uint4(0, 0, 0, 0);
                    if (w < words) {
                        x[u] = __ldcg(a + w);
                        y[u] = __ldcg(b + w);
                    }
                }
#pragma unroll
                for (int u = 0; u < kCmpUnroll; ++u)
                    diff |= (x[u].x ^ y[u].x) | (x[u].y ^ y[u].y) | (x[u].z ^ y[u].z) | (x[u].w ^ y[u].w);
            }
            v = __any_sync(0xffffffffu, diff != 0) ? PK_PAGE_DIFFERS : PK_PAGE_EQUAL;
        }
        if (lane == 0) {
            verdict[j] = v;
            atomicAdd_block(&block_counts[v], 1ull);
        }
    }
    pk::pdl_launch_dependents();
    __syncthreads();
    if (threadIdx.x < 3 && block_counts[threadIdx.x]) atomicAdd(&counts[threadIdx.x], block_counts[threadIdx.x]);
}

}  // namespace

cudaError_t pk_launch_compare_pages(const uint32_t *slots, const uint8_t *pages, const uint8_t *ref_pages, uint64_t n,
                                    uint64_t n_ref, uint64_t page_bytes, int32_t *verdict, unsigned long long *counts,
                                    int32_t *status, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const uint64_t blocks = (n + kCmpThreads / 32 - 1) / (kCmpThreads / 32);
    const cudaError_t e = pk_launch(k_compare_pages, (unsigned)blocks, kCmpThreads, s, slots, pages, ref_pages, n,
                                    n_ref, page_bytes, verdict, counts, status);
    return e != cudaSuccess ? e : cudaGetLastError();
}
