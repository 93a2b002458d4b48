// pk_internal.h -- context, table entry layout and kernel launchers of libpk.
#pragma once
#include <cuda_runtime_api.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/pk.h"

// One table entry, 32 bytes (one DRAM sector):
//   k[0..3]  the 16-byte key prefix, stored byte for byte (all zero = empty)
//   slot     the chunk slot bound to the key
//   owner    during a store call: ~(lowest entry index that claimed the key)
//   epoch    number of the store call that inserted the key (0 while empty)
struct alignas(32) pk_entry {
    uint32_t k[4];
    uint32_t slot;   // slot and owner form one little-endian 64-bit word
    uint32_t owner;  // (owner in the high half), raised by atomicMax
    unsigned long long epoch;
};
static_assert(sizeof(pk_entry) == PK_ENTRY_BYTES, "entry layout");
static_assert(offsetof(pk_entry, owner) == offsetof(pk_entry, slot) + 4 && offsetof(pk_entry, slot) % 8 == 0,
              "slot and owner form one 64-bit word");

struct pk_ctx {
    uint32_t chunk_tokens;
    uint32_t capacity_log2;
    uint32_t max_probe;
    uint64_t capacity;
    pk_entry *table;
    unsigned long long *counter_dev;  // [0] entries in the table; [1] requests handed out by a lookup-and-store;
                                      // [2] entries deferred in a store call; [3], [4] keys its claims and its
                                      // admission pass claimed (folded into [0] by its finalize kernel); [5] CTAs
                                      // of its claim kernel done
    unsigned long long epoch;         // last store call number
    unsigned long long *stamps;       // budget mode: last-use stamp per entry (pk_attach_stamps), else NULL
    uint32_t pad_kw[64];              // K_t + W_t of a chunk's final (padding-only) block, C % 16 == 0
    uint32_t sm_count;                // SMs of the context's device (0 if unknown): picks the round form
};

// internal per-entry states between the store kernels (never returned)
#define PK_STORE_PENDING 0x40000000   /* claimed or bid: the finalize kernel decides */
#define PK_STORE_DEFERRED 0x40000001  /* absent, left to the admission pass */

// Launchers (pk_derive.cu, pk_table.cu).  Each returns the launch error.
cudaError_t pk_launch_digest_descriptors(const uint8_t *enc, uint64_t enc_bytes, const int64_t *enc_off,
                                         uint32_t D, uint8_t *digests, int32_t *status, cudaStream_t s);
cudaError_t pk_launch_derive(const pk_ctx *ctx, const int32_t *tokens, uint64_t n_tokens,
                             const int64_t *tok_off, uint32_t R, const uint32_t *desc_idx,
                             const uint8_t *digests, uint32_t D, int64_t *key_off, uint8_t *keys,
                             uint64_t key_capacity, int32_t *status, cudaStream_t s);
cudaError_t pk_launch_derive_enc(const pk_ctx *ctx, const int32_t *tokens, uint64_t n_tokens,
                                 const int64_t *tok_off, uint32_t R, const uint32_t *desc_idx, const uint8_t *enc,
                                 uint64_t enc_bytes, const int64_t *enc_off, uint32_t D, uint8_t *digests,
                                 int64_t *key_off, uint8_t *keys, uint64_t key_capacity, int32_t *status,
                                 cudaStream_t s);
cudaError_t pk_launch_lookup(const pk_ctx *ctx, const uint8_t *keys, const int64_t *key_off, uint32_t R,
                             uint64_t key_capacity, int32_t *hit_chunks, uint32_t *slots, int32_t *status,
                             cudaStream_t s);
cudaError_t pk_launch_store_noalloc(pk_entry *table, uint32_t capacity_log2, uint32_t max_probe,
                                    const uint8_t *keys, const uint32_t *slots, uint64_t n, const int64_t *key_off,
                                    const int32_t *hit_chunks, uint32_t R, int32_t *result, uint32_t *slot_out,
                                    int32_t *status, cudaStream_t s);
cudaError_t pk_launch_mark_loaded(const pk_ctx *ctx, cudaStream_t s);
cudaError_t pk_launch_load_table(const pk_ctx *ctx, const void *src, cudaStream_t s);
cudaError_t pk_launch_store(const pk_ctx *ctx, unsigned long long epoch, const uint8_t *keys,
                            const uint32_t *slots, uint64_t n, const int64_t *key_off,
                            const int32_t *hit_chunks, uint32_t R, int32_t *result, uint32_t *slot_out,
                            int32_t *status, cudaStream_t s);
uint64_t pk_content_scratch_bytes_impl(uint64_t n_bytes);
cudaError_t pk_launch_content_digest(const uint8_t *bytes, uint64_t n_bytes, uint8_t *scratch, uint8_t *top,
                                     cudaStream_t s);
cudaError_t pk_launch_content_digests(const uint8_t *const *bytes, const uint64_t *n_bytes, uint32_t n,
                                      uint8_t *scratch, const uint64_t *scratch_off, uint8_t *tops, cudaStream_t s);
cudaError_t pk_launch_compare_pages(const uint32_t *slots, const uint8_t *pages, const uint8_t *ref_pages, uint64_t n,
                                    uint64_t n_ref, uint64_t page_bytes, int32_t *verdict, unsigned long long *counts,
                                    int32_t *status, cudaStream_t s);
uint64_t pk_evict_scratch_bytes_impl(uint64_t capacity);
// spin_limit: polls of a barrier wait before it gives up (0 = the default of
// about a second); withhold_first_cta: CTA 0 does not arrive at the first
// barrier (the timeout test).
cudaError_t pk_launch_evict(const pk_ctx *ctx, uint64_t budget, uint64_t keep, void *scratch, uint32_t *evicted,
                            uint64_t evicted_cap, unsigned long long *n_evicted, int32_t *status, cudaStream_t s,
                            uint32_t spin_limit = 0, bool withhold_first_cta = false);
cudaError_t pk_launch_key_strings(const uint8_t *keys, uint64_t n, const uint8_t *prefix, uint32_t plen,
                                  uint32_t width, uint8_t *out, cudaStream_t s);
cudaError_t pk_launch_lookup_store(const pk_ctx *ctx, unsigned long long epoch, const uint8_t *keys,
                                   const uint32_t *new_slots, const int64_t *key_off, uint32_t R,
                                   uint64_t key_capacity, int32_t *hit_chunks, uint32_t *slots, int32_t *result,
                                   uint32_t *slot_out, int32_t *status, cudaStream_t s);

#if defined(__CUDACC__)
#include <utility>
// Launch with programmatic stream serialization (see pk_device.cuh).
template <typename... KArgs, typename... Args>
static inline cudaError_t pk_launch(void (*kernel)(KArgs...), unsigned grid, unsigned block, cudaStream_t s,
                                    Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
// The same with dynamic shared memory.
template <typename... KArgs, typename... Args>
static inline cudaError_t pk_launch_smem(void (*kernel)(KArgs...), unsigned grid, unsigned block, size_t smem,
                                         cudaStream_t s, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
#endif
