// pk_derive.cu -- key derivation kernels (sm_103a).
//
//   descriptor digests  d_j = SHA-256(enc_j)                       (Eq. 3, H over enc)
//   chunk offsets       key_off = exclusive scan of floor(T_r / C)  (full chunks only, Sec. 4.4)
//   chunk digests       c_i = SHA-256(LE int32 tokens of chunk i)  (the content part of f(x, .))
//   chain               k_i = SHA-256(k_{i-1} || d || c_i)         (the digest folded into every key)
//
// SHA-256 is plain 32-bit integer work: funnel-shift rotates, 3-input logic
// and 3-input adds, no tensor cores.  The chunk digests are fully parallel
// (one thread per chunk, message words in registers, 128-bit token loads when
// the chunk start is 16-byte aligned); the chain is serial per request (one
// thread per request).  The chunk digests are staged in the output key buffer
// and overwritten in place by the chain, so derivation needs no scratch memory.
#include <cuda_runtime.h>

#include "pk_device.cuh"
#include "pk_internal.h"
#include "pk_sha256.cuh"

namespace {

using pk::set_status;

// ---------------------------------------------------------------------------
// Descriptor digests: one thread per descriptor.
// ---------------------------------------------------------------------------
__global__ void k_digest_descriptors(const uint8_t *__restrict__ enc, uint64_t enc_bytes,
                                     const int64_t *__restrict__ enc_off, uint32_t D,
                                     uint8_t *__restrict__ digests, int32_t *status) {
    const uint32_t j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= D) return;
    const int64_t a = enc_off[j], b = enc_off[j + 1];
    if (a < 0 || b < a || (uint64_t)b > enc_bytes) {
        set_status(status, PK_ERR_ARG);
        return;
    }
    pk::sha256_bytes(enc + a, (uint64_t)(b - a), digests + 32ull * j);
}

// ---------------------------------------------------------------------------
// Chunk offsets: one block.  Validates the request layout, then writes the
// exclusive scan of floor(T_r / C).  Any invalid request zeroes all offsets.
// ---------------------------------------------------------------------------
constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads)
k_chunk_offsets(const int64_t *__restrict__ tok_off, uint32_t R, uint64_t n_tokens, uint32_t C,
                const uint32_t *__restrict__ desc_idx, uint32_t D, uint64_t key_capacity,
                int64_t *__restrict__ key_off, int32_t *status) {
    __shared__ long long warp_sums[kScanThreads / 32];
    __shared__ long long total_s;
    const uint32_t tid = threadIdx.x;
    const uint64_t per = (R + kScanThreads - 1) / kScanThreads;
    const uint64_t lo = tid * per;
    const uint64_t hi = lo + per < R ? lo + per : R;

    bool bad = false;
    long long local = 0;
    for (uint64_t r = lo; r < hi; ++r) {
        const int64_t a = tok_off[r], b = tok_off[r + 1];
        if (a < 0 || b < a || (uint64_t)b > n_tokens || desc_idx[r] >= D) bad = true;
        else local += (b - a) / C;
    }
    bad = __syncthreads_or(bad);

    // block exclusive scan of the per-thread sums
    const int lane = tid & 31, warp = tid >> 5;
    long long incl = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
    }
    if (lane == 31) warp_sums[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        long long ws = warp_sums[lane];
        long long wincl = ws;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const long long v = __shfl_up_sync(0xffffffffu, wincl, o);
            if (lane >= o) wincl += v;
        }
        warp_sums[lane] = wincl - ws;
        if (lane == 31) total_s = wincl;
    }
    __syncthreads();
    long long run = warp_sums[warp] + incl - local;
    const bool too_many = (unsigned long long)total_s > key_capacity;

    if (tid == 0) key_off[0] = 0;
    if (bad || too_many) {
        for (uint64_t r = lo; r < hi; ++r) key_off[r + 1] = 0;
        if (tid == 0) set_status(status, PK_ERR_ARG);
        return;
    }
    for (uint64_t r = lo; r < hi; ++r) {
        run += (tok_off[r + 1] - tok_off[r]) / C;
        key_off[r + 1] = run;
    }
}

__device__ __forceinline__ void store_digest(uint8_t *dst, const uint32_t st[8]) {
    uint4 *q = reinterpret_cast<uint4 *>(dst);
    q[0] = make_uint4(pk::bswap32(st[0]), pk::bswap32(st[1]), pk::bswap32(st[2]), pk::bswap32(st[3]));
    q[1] = make_uint4(pk::bswap32(st[4]), pk::bswap32(st[5]), pk::bswap32(st[6]), pk::bswap32(st[7]));
}

// 16 message words of one 64-byte block of int32 tokens (little-endian bytes,
// read by SHA-256 as big-endian words).
__device__ __forceinline__ void load_block(const int32_t *__restrict__ src, bool aligned, uint32_t w[16]) {
    if (aligned) {
        const uint4 *q = reinterpret_cast<const uint4 *>(src);
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const uint4 x = __ldg(q + v);
            w[4 * v + 0] = pk::bswap32(x.x);
            w[4 * v + 1] = pk::bswap32(x.y);
            w[4 * v + 2] = pk::bswap32(x.z);
            w[4 * v + 3] = pk::bswap32(x.w);
        }
    } else {
#pragma unroll
        for (int t = 0; t < 16; ++t) w[t] = pk::bswap32((uint32_t)__ldg(src + t));
    }
}

// ---------------------------------------------------------------------------
// Chunk digests: one thread per chunk, 32 consecutive chunks per warp.  CT > 0
// fixes the chunk size at compile time (the padding block is then a constant
// message whose schedule the compiler folds); CT == 0 takes it at run time.
// The next 64-byte block is loaded while the current one is compressed.
// ---------------------------------------------------------------------------
template <int CT>
__global__ void __launch_bounds__(128)
k_chunk_digest(const int32_t *__restrict__ tokens, const int64_t *__restrict__ tok_off,
               const int64_t *__restrict__ key_off, uint32_t R, uint32_t C_rt,
               uint8_t *__restrict__ keys) {
    if (R == 0) return;
    const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t g0 = g - (threadIdx.x & 31);
    const int64_t total = __ldg(key_off + R);
    if (g0 >= total) return;  // whole warp past the end
    const uint32_t r = pk::lane_request(key_off, R, g0, total, g);
    if (g >= total) return;
    const int64_t i = g - __ldg(key_off + r);
    const uint32_t C = CT > 0 ? (uint32_t)CT : C_rt;
    const int32_t *src = tokens + __ldg(tok_off + r) + i * (int64_t)C;
    const bool aligned = (reinterpret_cast<uintptr_t>(src) & 15) == 0;

    uint32_t st[8];
    pk::init_state(st);
    const uint32_t nfull = C / 16;
    uint32_t w[16];
    if (nfull > 0) load_block(src, aligned, w);
#pragma unroll 1
    for (uint32_t b = 0; b < nfull; ++b) {
        uint32_t nx[16];
        if (b + 1 < nfull) load_block(src + 16 * (b + 1), aligned, nx);
        pk::compress16(st, w);
#pragma unroll
        for (int t = 0; t < 16; ++t) w[t] = nx[t];
    }
    const uint64_t bits = (uint64_t)C * 32u;
    const int rem = (int)(C % 16);
    if (rem == 0) {
        pk::compress(st, 0x80000000u, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0,
                     (uint32_t)(bits >> 32), (uint32_t)bits);
    } else {
        const int32_t *tail = src + 16 * nfull;
#pragma unroll
        for (int t = 0; t < 16; ++t)
            w[t] = t < rem ? pk::bswap32((uint32_t)__ldg(tail + t)) : (t == rem ? 0x80000000u : 0u);
        if (rem <= 13) {
            w[14] = (uint32_t)(bits >> 32);
            w[15] = (uint32_t)bits;
            pk::compress16(st, w);
        } else {
            pk::compress16(st, w);
            pk::compress(st, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0,
                         (uint32_t)(bits >> 32), (uint32_t)bits);
        }
    }
    store_digest(keys + 32 * g, st);
}

// ---------------------------------------------------------------------------
// Chain: one thread per request.  Message = k_{i-1} || d (block 1) then
// c_i || padding for a 96-byte message (block 2, constant tail).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(64)
k_chain(const int64_t *__restrict__ key_off, const uint32_t *__restrict__ desc_idx,
        const uint8_t *__restrict__ digests, uint32_t R, uint32_t D, uint8_t *keys) {
    const uint32_t r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= R) return;
    const int64_t a = key_off[r];
    const int64_t n = key_off[r + 1] - a;
    const uint32_t di = desc_idx[r];
    if (n <= 0 || di >= D) return;

    const uint4 *dq = reinterpret_cast<const uint4 *>(digests + 32ull * di);
    const uint4 d_lo = __ldg(dq), d_hi = __ldg(dq + 1);
    const uint32_t d0 = pk::bswap32(d_lo.x), d1 = pk::bswap32(d_lo.y), d2 = pk::bswap32(d_lo.z),
                   d3 = pk::bswap32(d_lo.w), d4 = pk::bswap32(d_hi.x), d5 = pk::bswap32(d_hi.y),
                   d6 = pk::bswap32(d_hi.z), d7 = pk::bswap32(d_hi.w);

    uint4 *kq = reinterpret_cast<uint4 *>(keys + 32ull * a);
    uint32_t p[8] = {0, 0, 0, 0, 0, 0, 0, 0};  // k_{-1} = 0^32
    uint4 c_lo = kq[0], c_hi = kq[1];
#pragma unroll 1
    for (int64_t i = 0; i < n; ++i) {
        uint4 n_lo = c_lo, n_hi = c_hi;
        if (i + 1 < n) {  // prefetch c_{i+1}
            n_lo = kq[2 * (i + 1)];
            n_hi = kq[2 * (i + 1) + 1];
        }
        uint32_t st[8];
        pk::init_state(st);
        pk::compress(st, p[0], p[1], p[2], p[3], p[4], p[5], p[6], p[7], d0, d1, d2, d3, d4, d5, d6, d7);
        pk::compress(st, pk::bswap32(c_lo.x), pk::bswap32(c_lo.y), pk::bswap32(c_lo.z), pk::bswap32(c_lo.w),
                     pk::bswap32(c_hi.x), pk::bswap32(c_hi.y), pk::bswap32(c_hi.z), pk::bswap32(c_hi.w),
                     0x80000000u, 0, 0, 0, 0, 0, 0, 96u * 8u);
#pragma unroll
        for (int j = 0; j < 8; ++j) p[j] = st[j];
        store_digest(keys + 32ull * (a + i), st);
        c_lo = n_lo;
        c_hi = n_hi;
    }
}

unsigned grid_for(uint64_t n, unsigned block) { return (unsigned)((n + block - 1) / block); }

}  // namespace

cudaError_t pk_launch_digest_descriptors(const uint8_t *enc, uint64_t enc_bytes, const int64_t *enc_off,
                                         uint32_t D, uint8_t *digests, int32_t *status, cudaStream_t s) {
    if (D == 0) return cudaSuccess;
    k_digest_descriptors<<<grid_for(D, 64), 64, 0, s>>>(enc, enc_bytes, enc_off, D, digests, status);
    return cudaGetLastError();
}

cudaError_t pk_launch_derive(const pk_ctx *ctx, const int32_t *tokens, uint64_t n_tokens,
                             const int64_t *tok_off, uint32_t R, const uint32_t *desc_idx,
                             const uint8_t *digests, uint32_t D, int64_t *key_off, uint8_t *keys,
                             uint64_t key_capacity, int32_t *status, cudaStream_t s) {
    const uint32_t C = ctx->chunk_tokens;
    k_chunk_offsets<<<1, kScanThreads, 0, s>>>(tok_off, R, n_tokens, C, desc_idx, D, key_capacity, key_off,
                                               status);
    if (R == 0 || key_capacity == 0) return cudaGetLastError();
    constexpr unsigned kDigestBlock = 64;
    const unsigned grid = grid_for(key_capacity, kDigestBlock);
    if (C == 256)
        k_chunk_digest<256><<<grid, kDigestBlock, 0, s>>>(tokens, tok_off, key_off, R, C, keys);
    else if (C == 16)
        k_chunk_digest<16><<<grid, kDigestBlock, 0, s>>>(tokens, tok_off, key_off, R, C, keys);
    else
        k_chunk_digest<0><<<grid, kDigestBlock, 0, s>>>(tokens, tok_off, key_off, R, C, keys);
    constexpr unsigned kChainBlock = 32;
    k_chain<<<grid_for(R, kChainBlock), kChainBlock, 0, s>>>(key_off, desc_idx, digests, R, D, keys);
    return cudaGetLastError();
}
