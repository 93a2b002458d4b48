// pk_content.cu -- content identity of large byte buffers (adapter tensors,
// checkpoints) on the GPU.  The paper binds an adapter by an identity of its
// contents (Sec. 5.3, request-level tags: every tensor's name, dtype, shape
// and bytes with the meaningful configuration fields) and leaves the identity
// function open as long as it is injective and stable (Sec. 5.1).  A single
// SHA-256 stream over a tensor is serial; this file computes a fixed-shape
// tree of SHA-256 instead: every level hashes each 1 KiB block of the level
// below (the last block zero-padded), until one 32-byte digest remains.  The
// shape depends only on the byte length, which the tensor identity binds
// (pk_tensor_identity), so the tree is injective wherever SHA-256 is.
#include <cuda_runtime.h>

#include "pk_device.cuh"
#include "pk_internal.h"
#include "pk_sha256.cuh"

namespace {

constexpr int kTreeThreads = 128;
constexpr uint64_t kTreeBlock = 1024;  // bytes per tree block

// 16 big-endian message words of bytes [off, off + 64) of src, zero past n.
__device__ __forceinline__ void load_words(const uint8_t *src, uint64_t n, uint64_t off, uint32_t w[16]) {
#pragma unroll
    for (int v = 0; v < 4; ++v) {
        const uint64_t o = off + 16 * v;
        uint4 x = make_uint4(0, 0, 0, 0);
        if (o + 16 <= n) {
            x = __ldcg(reinterpret_cast<const uint4 *>(src + o));
        } else if (o < n) {  // the buffer's last partial 16 bytes
            uint32_t b[4] = {0, 0, 0, 0};
            for (uint64_t k = o; k < n; ++k) b[(k - o) / 4] |= (uint32_t)src[k] << (8 * ((k - o) % 4));
            x = make_uint4(b[0], b[1], b[2], b[3]);
        }
        w[4 * v + 0] = pk::bswap32(x.x);
        w[4 * v + 1] = pk::bswap32(x.y);
        w[4 * v + 2] = pk::bswap32(x.z);
        w[4 * v + 3] = pk::bswap32(x.w);
    }
}

// dst[t] = SHA-256 of block t (1 KiB) of src[0, n), zero-padded, t < m.
__global__ void __launch_bounds__(kTreeThreads)
k_tree_level(const uint8_t *src, uint64_t n, uint8_t *dst, uint64_t m) {
    __shared__ uint32_t sK[64];
    if (threadIdx.x < 64) sK[threadIdx.x] = pk::kSha256K[threadIdx.x];
    __syncthreads();
    pk::pdl_wait(src, dst);
    const uint64_t t = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t < m) {
        uint32_t st[8], w[16];
        pk::init_state(st);
        const uint64_t base = t * kTreeBlock;
#pragma unroll 1
        for (uint64_t b = 0; b < kTreeBlock / 64; ++b) {
            load_words(src, n, base + 64 * b, w);
            pk::compress_rolled(st, w, sK);
        }
        // padding of a 1024-byte message: 0x80, zeros, the length in bits (8192)
#pragma unroll
        for (int k = 0; k < 16; ++k) w[k] = 0;
        w[0] = 0x80000000u;
        w[15] = (uint32_t)(kTreeBlock * 8);
        pk::compress_rolled(st, w, sK);
        uint4 *q = reinterpret_cast<uint4 *>(dst + 32 * t);
        q[0] = make_uint4(pk::bswap32(st[0]), pk::bswap32(st[1]), pk::bswap32(st[2]), pk::bswap32(st[3]));
        q[1] = make_uint4(pk::bswap32(st[4]), pk::bswap32(st[5]), pk::bswap32(st[6]), pk::bswap32(st[7]));
    }
    pk::pdl_launch_dependents();
}

uint64_t blocks_of(uint64_t n) { return n == 0 ? 1 : (n + kTreeBlock - 1) / kTreeBlock; }

}  // namespace

uint64_t pk_content_scratch_bytes_impl(uint64_t n_bytes) {
    uint64_t total = 0, m = blocks_of(n_bytes);
    while (true) {
        total += 32 * m;
        if (m == 1) break;
        m = blocks_of(32 * m);
    }
    return total;
}

cudaError_t pk_launch_content_digest(const uint8_t *bytes, uint64_t n_bytes, uint8_t *scratch, uint8_t *top,
                                     cudaStream_t s) {
    const uint8_t *src = bytes;
    uint64_t n = n_bytes, m = blocks_of(n_bytes);
    uint8_t *dst = scratch;
    while (true) {
        uint8_t *out = m == 1 ? top : dst;
        const cudaError_t e = pk_launch(k_tree_level, (unsigned)((m + kTreeThreads - 1) / kTreeThreads),
                                        kTreeThreads, s, src, n, out, m);
        if (e != cudaSuccess) return e;
        if (m == 1) break;
        src = dst;
        n = 32 * m;
        dst += 32 * m;
        m = blocks_of(n);
    }
    return cudaGetLastError();
}
