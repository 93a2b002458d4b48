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

#include <mutex>

#include "pk_device.cuh"
#include "pk_internal.h"
#include "pk_sha256.cuh"

namespace {

constexpr int kTreeThreads = 128;
constexpr uint64_t kTreeBlock = 1024;  // bytes per tree block

// 16-byte L2 load kept in program order (a prefetch the compiler must not sink).
__device__ __forceinline__ uint4 ld_cg_v4_ordered(const void *p) {
    uint4 v;
    asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// 16 big-endian message words of bytes [off, off + 64) of src, zero past n.
__device__ __forceinline__ void load_words(const uint8_t *src, uint64_t n, uint64_t off, uint32_t w[16]) {
#pragma unroll
    for (int v = 0; v < 4; ++v) {
        const uint64_t o = off + 16 * v;
        uint4 x = make_uint4(0, 0, 0, 0);
        if (o + 16 <= n) {
            x = ld_cg_v4_ordered(src + o);
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

// One tree level of up to kMaxSeg buffers in one launch: segment j hashes the
// 1 KiB blocks of src[0, n) (zero-padded) into dst, its blocks being the
// launch's threads first[j] .. first[j+1]-1 (the segments passed by value stay
// within the 4 KiB kernel-parameter space).
constexpr uint32_t kMaxSeg = 128;
struct TreeSeg {
    const uint8_t *src;
    uint64_t n;
    uint8_t *dst;
};
struct TreeLevel {
    uint32_t count;
    uint32_t first[kMaxSeg + 1];  // first[count] = threads of the launch
    TreeSeg seg[kMaxSeg];
};
static_assert(sizeof(TreeLevel) <= 4000, "kernel parameter space");

// K_t + W_t of the final block of every 1 KiB message: 0x80, zeros, the length in bits (8192).
struct PadKW1K {
    uint32_t kw[64];
};

// F is the round form of pk_sha256.cuh (kAddsFma for levels of many blocks);
// `one` is its run-time constant 1.
template <int F>
__global__ void __launch_bounds__(kTreeThreads)
k_tree_level(const __grid_constant__ TreeLevel lv, const __grid_constant__ PadKW1K pad, uint32_t one) {
    __shared__ uint32_t sK[64], sPad[64];
    if (threadIdx.x < 64) {
        sK[threadIdx.x] = pk::kSha256K[threadIdx.x];
        sPad[threadIdx.x] = pad.kw[threadIdx.x];
    }
    __syncthreads();
    pk::pdl_wait();
    const uint64_t t = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t < lv.first[lv.count]) {
        uint32_t lo = 0, hi = lv.count;  // first[lo] <= t < first[hi]
        while (hi - lo > 1) {
            const uint32_t mid = (lo + hi) >> 1;
            if (lv.first[mid] <= t) lo = mid; else hi = mid;
        }
        const TreeSeg sg = lv.seg[lo];
        const uint64_t b = t - lv.first[lo];
        uint32_t st[8], w[16], wn[16];
        pk::init_state(st);
        const uint64_t base = b * kTreeBlock;
        load_words(sg.src, sg.n, base, wn);
#pragma unroll 1
        for (uint64_t q = 0; q < kTreeBlock / 64; ++q) {  // the next 64 bytes load while these are compressed
#pragma unroll
            for (int k = 0; k < 16; ++k) w[k] = wn[k];
            if (q + 1 < kTreeBlock / 64) load_words(sg.src, sg.n, base + 64 * (q + 1), wn);
            pk::compress_rolled<F>(st, w, sK, one);
        }
        pk::compress_kw<F>(st, sPad, one);  // the padding block, rounds only
        uint4 *q = reinterpret_cast<uint4 *>(sg.dst + 32 * b);
        q[0] = make_uint4(pk::bswap32(st[0]), pk::bswap32(st[1]), pk::bswap32(st[2]), pk::bswap32(st[3]));
        q[1] = make_uint4(pk::bswap32(st[4]), pk::bswap32(st[5]), pk::bswap32(st[6]), pk::bswap32(st[7]));
    }
    pk::pdl_launch_dependents();
}

uint64_t blocks_of(uint64_t n) { return n == 0 ? 1 : (n + kTreeBlock - 1) / kTreeBlock; }

// Threads of a level from which the multiply-add round form is used (3 warps
// per SM sub-partition, as for the chunk digests), computed once per device;
// 0 (never) if the device cannot be queried.
uint64_t fma_threshold() {
    static std::mutex mu;
    static uint64_t cache[256] = {};
    static bool known[256] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) return 0;
    std::lock_guard<std::mutex> lock(mu);
    if (!known[dev]) {
        int sms = 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && sms > 0)
            cache[dev] = 3ull * 4 * 32 * (uint64_t)sms;
        known[dev] = true;
    }
    return cache[dev];
}

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

// Tree tops of n buffers: every level of every buffer not yet reduced to one
// digest in one launch per level (kMaxSeg buffers at a time).  Buffer j's
// levels go to scratch at scratch_off[j]; its last level writes tops[32 j].
cudaError_t pk_launch_content_digests(const uint8_t *const *bytes, const uint64_t *n_bytes, uint32_t n,
                                      uint8_t *scratch, const uint64_t *scratch_off, uint8_t *tops, cudaStream_t s) {
    PadKW1K pad;
    {
        const uint32_t m[16] = {0x80000000u, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, (uint32_t)(kTreeBlock * 8)};
        pk::kw_table(m, pad.kw);
    }
    const uint64_t fma_from = fma_threshold();
    const uint32_t one = 1u;
    for (uint32_t j0 = 0; j0 < n; j0 += kMaxSeg) {
        const uint32_t cnt = n - j0 < kMaxSeg ? n - j0 : kMaxSeg;
        TreeSeg cur[kMaxSeg];
        uint64_t m[kMaxSeg];
        bool done[kMaxSeg];
        for (uint32_t j = 0; j < cnt; ++j) {
            cur[j] = TreeSeg{bytes[j0 + j], n_bytes[j0 + j], scratch + scratch_off[j0 + j]};
            m[j] = blocks_of(n_bytes[j0 + j]);
            done[j] = false;
        }
        for (;;) {
            TreeLevel lv;
            lv.count = 0;
            uint64_t threads = 0;
            for (uint32_t j = 0; j < cnt; ++j) {
                if (done[j]) continue;
                TreeSeg sg = cur[j];
                if (m[j] == 1) sg.dst = tops + 32ull * (j0 + j);
                lv.first[lv.count] = (uint32_t)threads;
                lv.seg[lv.count++] = sg;
                threads += m[j];
            }
            if (lv.count == 0) break;
            if (threads >= (1ull << 31)) return cudaErrorInvalidValue;
            lv.first[lv.count] = (uint32_t)threads;
            const unsigned grid = (unsigned)((threads + kTreeThreads - 1) / kTreeThreads);
            const cudaError_t e = fma_from && threads >= fma_from
                                      ? pk_launch(k_tree_level<pk::kAddsFma>, grid, kTreeThreads, s, lv, pad, one)
                                      : pk_launch(k_tree_level<pk::kAddsPlain>, grid, kTreeThreads, s, lv, pad, one);
            if (e != cudaSuccess) return e;
            for (uint32_t j = 0; j < cnt; ++j) {  // the next level reads this one
                if (done[j]) continue;
                if (m[j] == 1) {
                    done[j] = true;
                    continue;
                }
                cur[j].src = cur[j].dst;
                cur[j].n = 32 * m[j];
                cur[j].dst += 32 * m[j];
                m[j] = blocks_of(cur[j].n);
            }
        }
    }
    return cudaGetLastError();
}

cudaError_t pk_launch_content_digest(const uint8_t *bytes, uint64_t n_bytes, uint8_t *scratch, uint8_t *top,
                                     cudaStream_t s) {
    const uint64_t off = 0;
    return pk_launch_content_digests(&bytes, &n_bytes, 1, scratch, &off, top, s);
}
