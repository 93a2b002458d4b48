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

#include <mutex>

#include "pk_device.cuh"
#include "pk_internal.h"
#include "pk_sha256.cuh"

namespace {

using pk::set_status;

// ---------------------------------------------------------------------------
// Descriptor digests: one warp per descriptor.  The warp copies the encoding
// into shared memory with coalesced byte loads (32 bytes per round trip), then
// one lane hashes it.  Encodings longer than the staging area are hashed from
// global memory.
// ---------------------------------------------------------------------------
constexpr int kDescWarps = 4;
constexpr int kDescStage = 2048;

// Warp `warp` of the calling block hashes descriptor j (all 32 lanes call).
__device__ __forceinline__ void hash_descriptor(uint8_t *stage, const uint8_t *enc, uint64_t enc_bytes,
                                                const int64_t *enc_off, uint32_t j,
                                                uint8_t *digests, int32_t *status) {
    const uint32_t lane = threadIdx.x & 31;
    const int64_t a = __ldcg(enc_off + j), b = __ldcg(enc_off + j + 1);
    if (a < 0 || b < a || (uint64_t)b > enc_bytes) {
        if (lane == 0) set_status(status, PK_ERR_ARG);
        return;
    }
    const int64_t len = b - a;
    const bool staged = len <= kDescStage;
    if (staged) {
#pragma unroll 4
        for (int64_t i = lane; i < len; i += 32) stage[i] = __ldcg(enc + a + i);
    }
    __syncwarp();
    if (lane == 0) pk::sha256_bytes(staged ? stage : enc + a, (uint64_t)len, digests + 32ull * j);
}

__global__ void __launch_bounds__(32 * kDescWarps)
k_digest_descriptors(const uint8_t *enc, uint64_t enc_bytes, const int64_t *enc_off,
                     uint32_t D, uint8_t *digests, int32_t *status) {
    __shared__ __align__(16) uint8_t stage[kDescWarps][kDescStage];
    pk::pdl_launch_dependents();
    pk::pdl_wait(enc, enc_off, digests, status);
    const uint32_t warp = threadIdx.x >> 5;
    const uint32_t j = blockIdx.x * kDescWarps + warp;
    if (j < D) hash_descriptor(stage[warp], enc, enc_bytes, enc_off, j, digests, status);
}

// ---------------------------------------------------------------------------
// Chunk offsets: one block, requests in tiles of kScanThreads * kScanItems.
// Each thread takes kScanItems consecutive requests of the tile (coalesced
// offset loads), the block scans the per-thread sums, and a running carry
// links the tiles.  Any invalid request (offsets decreasing, negative or past
// n_tokens, descriptor index >= D) or a total above key_capacity zeroes all
// offsets afterwards and reports PK_ERR_ARG.
// ---------------------------------------------------------------------------
constexpr int kScanThreads = 1024;
constexpr int kScanItems = 4;

__global__ void __launch_bounds__(kScanThreads)
k_chunk_offsets(const int64_t *tok_off, uint32_t R, uint64_t n_tokens, uint32_t C,
                const uint32_t *desc_idx, uint32_t D, uint64_t key_capacity,
                int64_t *key_off, int32_t *status) {
    __shared__ long long warp_sums[kScanThreads / 32];
    __shared__ long long tile_total;
    pk::pdl_launch_dependents();
    pk::pdl_wait(tok_off, desc_idx, key_off, status);
    const uint32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) key_off[0] = 0;
    bool bad = false;
    long long carry = 0;
    // a tile's inputs (its threads' tok_off[r0 .. r0 + kScanItems], desc_idx[r0 .. r0 + kScanItems)) are loaded
    // one tile ahead, so that they are in flight during the previous tile's scan
    constexpr uint64_t kTile = (uint64_t)kScanThreads * kScanItems;
    int64_t to_cur[kScanItems + 1], to_nxt[kScanItems + 1] = {};
    uint32_t di_cur[kScanItems], di_nxt[kScanItems] = {};
    auto load_tile = [&](uint64_t base, int64_t *to, uint32_t *di) {
        const uint64_t r0 = base + (uint64_t)tid * kScanItems;
#pragma unroll
        for (int j = 0; j <= kScanItems; ++j) to[j] = r0 + j <= R ? tok_off[r0 + j] : 0;
#pragma unroll
        for (int j = 0; j < kScanItems; ++j) di[j] = r0 + j < R ? desc_idx[r0 + j] : 0u;
    };
    if (R > 0) load_tile(0, to_cur, di_cur);
    for (uint64_t base = 0; base < R; base += kTile) {
        if (base + kTile < R) load_tile(base + kTile, to_nxt, di_nxt);
        const uint64_t r0 = base + (uint64_t)tid * kScanItems;
        long long n[kScanItems];
        long long local = 0;
#pragma unroll
        for (int j = 0; j < kScanItems; ++j) {
            const uint64_t r = r0 + j;
            n[j] = 0;
            if (r < R) {
                const int64_t a = to_cur[j], b = to_cur[j + 1];
                if (a < 0 || b < a || (uint64_t)b > n_tokens || di_cur[j] >= D) {
                    bad = true;
                } else {  // 32-bit division when the request fits (64-bit division is a long library sequence)
                    const uint64_t len = (uint64_t)(b - a);
                    n[j] = len >> 32 ? (long long)(len / C) : (long long)((uint32_t)len / C);
                }
            }
            local += n[j];
        }
        // block exclusive scan of the per-thread sums
        long long incl = local;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const long long v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) warp_sums[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            const long long ws = warp_sums[lane];
            long long wincl = ws;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const long long v = __shfl_up_sync(0xffffffffu, wincl, o);
                if (lane >= o) wincl += v;
            }
            warp_sums[lane] = wincl - ws;
            if (lane == 31) tile_total = wincl;
        }
        __syncthreads();
        long long run = carry + warp_sums[warp] + incl - local;
#pragma unroll
        for (int j = 0; j < kScanItems; ++j) {
            if (r0 + j < R) {
                run += n[j];
                key_off[r0 + j + 1] = run;
            }
        }
        carry += tile_total;
        __syncthreads();  // warp_sums and tile_total are reused by the next tile
#pragma unroll
        for (int j = 0; j <= kScanItems; ++j) to_cur[j] = to_nxt[j];
#pragma unroll
        for (int j = 0; j < kScanItems; ++j) di_cur[j] = di_nxt[j];
    }
    bad = __syncthreads_or(bad);
    if (bad || (unsigned long long)carry > key_capacity) {
        for (uint64_t r = tid; r < R; r += kScanThreads) key_off[r + 1] = 0;
        if (tid == 0) set_status(status, PK_ERR_ARG);
    }
}

__device__ __forceinline__ void store_digest(uint8_t *dst, const uint32_t st[8]) {
    uint4 *q = reinterpret_cast<uint4 *>(dst);
    q[0] = make_uint4(pk::bswap32(st[0]), pk::bswap32(st[1]), pk::bswap32(st[2]), pk::bswap32(st[3]));
    q[1] = make_uint4(pk::bswap32(st[4]), pk::bswap32(st[5]), pk::bswap32(st[6]), pk::bswap32(st[7]));
}

// 16 message words of one 64-byte block of int32 tokens (little-endian bytes,
// read by SHA-256 as big-endian words), straight from global memory.
__device__ __forceinline__ void load_block_global(const int32_t *src, uint32_t w[16]) {
#pragma unroll
    for (int t = 0; t < 16; ++t) w[t] = pk::bswap32((uint32_t)__ldcg(src + t));
}

// Asynchronous 64-byte copy global -> shared (4 x 16 B; both 16-byte aligned).
__device__ __forceinline__ void cp_async_block(uint32_t *smem_dst, const int32_t *src) {
    const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem_dst);
#pragma unroll
    for (int v = 0; v < 4; ++v)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d + 16 * v), "l"(src + 4 * v) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Round constants and the padding block's schedule in shared memory.
struct PadKW {
    uint32_t kw[64];  // K_t + W_t of the final block of a message of 64k bytes (padding only)
};

__device__ __forceinline__ void load_tables(uint32_t *sK, uint32_t *sPad, const PadKW &pad) {
    for (int i = threadIdx.x; i < 64; i += blockDim.x) {
        sK[i] = pk::kSha256K[i];
        sPad[i] = pad.kw[i];
    }
}

// ---------------------------------------------------------------------------
// Chunk digests: one thread per chunk, 32 consecutive chunks per warp.  Token
// blocks are staged through a 3-deep shared-memory ring with cp.async, so the
// load of block b+2 overlaps the compression of block b.  For chunk sizes that
// are multiples of 16 tokens the final block is pure padding, identical for
// every chunk: it runs as rounds only on a schedule precomputed on the host.
// ---------------------------------------------------------------------------
constexpr int kDigestBlock = 128;
constexpr int kStages = 3;
constexpr uint32_t kFmaWarps = 3;  // warps of chunks per SM sub-partition from which kAddsFma is used

// c = SHA-256 of chunk g (request r), written to keys[g].  F is the round
// form (pk_sha256.cuh: kAddsFma when several warps share each sub-partition).
template <int F>
__device__ __forceinline__ void digest_chunk(const int32_t *tokens, const int64_t *tok_off,
                                             const int64_t *key_off, uint32_t r, int64_t g, uint32_t C,
                                             const uint32_t *sK, const uint32_t *sPad,
                                             uint32_t (*ring)[kDigestBlock][16], uint8_t *keys, uint32_t one) {
    const int64_t i = g - __ldcg(key_off + r);
    const int32_t *src = tokens + __ldcg(tok_off + r) + i * (int64_t)C;
    const bool aligned = (reinterpret_cast<uintptr_t>(src) & 15) == 0;

    uint32_t st[8];
    pk::init_state(st);
    const uint32_t nfull = C / 16;
    uint32_t w[16];
    if (aligned) {
#pragma unroll
        for (int b = 0; b < kStages - 1; ++b) {
            if ((uint32_t)b < nfull) cp_async_block(ring[b][threadIdx.x], src + 16 * b);
            cp_async_commit();
        }
#pragma unroll 1
        for (uint32_t b = 0; b < nfull; ++b) {
            const uint32_t ahead = b + kStages - 1;
            if (ahead < nfull) cp_async_block(ring[ahead % kStages][threadIdx.x], src + 16 * ahead);
            cp_async_commit();
            cp_async_wait<kStages - 1>();  // block b has landed
            const uint4 *q = reinterpret_cast<const uint4 *>(ring[b % kStages][threadIdx.x]);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                const uint4 x = q[v];
                w[4 * v + 0] = pk::bswap32(x.x);
                w[4 * v + 1] = pk::bswap32(x.y);
                w[4 * v + 2] = pk::bswap32(x.z);
                w[4 * v + 3] = pk::bswap32(x.w);
            }
            pk::compress_rolled<F>(st, w, sK, one);
        }
        cp_async_wait<0>();
    } else {
#pragma unroll 1
        for (uint32_t b = 0; b < nfull; ++b) {
            load_block_global(src + 16 * b, w);
            pk::compress_rolled<F>(st, w, sK, one);
        }
    }
    const uint64_t bits = (uint64_t)C * 32u;
    const int rem = (int)(C % 16);
    if (rem == 0) {
        pk::compress_kw<F>(st, sPad, one);
    } else {
        const int32_t *tail = src + 16 * nfull;
#pragma unroll
        for (int t = 0; t < 16; ++t)
            w[t] = t < rem ? pk::bswap32((uint32_t)__ldcg(tail + t)) : (t == rem ? 0x80000000u : 0u);
        if (rem <= 13) {
            w[14] = (uint32_t)(bits >> 32);
            w[15] = (uint32_t)bits;
            pk::compress_rolled<F>(st, w, sK, one);
        } else {
            pk::compress_rolled<F>(st, w, sK, one);
#pragma unroll
            for (int t = 0; t < 16; ++t) w[t] = 0;
            w[14] = (uint32_t)(bits >> 32);
            w[15] = (uint32_t)bits;
            pk::compress_rolled<F>(st, w, sK, one);
        }
    }
    store_digest(keys + 32 * g, st);
}

// Optional descriptor work for the same launch (fused a0): the first
// desc_blocks blocks hash descriptor encodings instead, one warp each.
struct DescWork {
    const uint8_t *enc;
    uint64_t enc_bytes;
    const int64_t *enc_off;
    uint32_t D;
    uint8_t *digests;
    int32_t *status;
    uint32_t desc_blocks;
};

// `one` is the run-time constant 1 of the multiply-add round form.
template <int F>
__global__ void __launch_bounds__(kDigestBlock)
k_chunk_digest(const int32_t *tokens, const int64_t *tok_off,
               const int64_t *key_off, uint32_t R, uint32_t C, const __grid_constant__ PadKW pad,
               uint8_t *keys, const __grid_constant__ DescWork dw, uint32_t one) {
    __shared__ uint32_t sK[64], sPad[64];
    __shared__ __align__(16) uint32_t ring[kStages][kDigestBlock][16];
    // The successor (the chain) is released as each block finishes, not at its start: released early,
    // its waiting CTAs, and those of the kernel after it, would sit on the SMs during the whole digest.
    if (blockIdx.x < dw.desc_blocks) {
        const uint8_t *enc = dw.enc;
        const int64_t *enc_off = dw.enc_off;
        uint8_t *digests = dw.digests;
        int32_t *dstatus = dw.status;
        pk::pdl_wait(enc, enc_off, digests, dstatus);
        const uint32_t warp = threadIdx.x >> 5;
        const uint32_t j = blockIdx.x * (kDigestBlock / 32) + warp;
        uint8_t *stage = reinterpret_cast<uint8_t *>(ring[0]) + warp * kDescStage;  // 4 x 2 KiB of the ring
        if (j < dw.D) hash_descriptor(stage, enc, dw.enc_bytes, enc_off, j, digests, dstatus);
        pk::pdl_launch_dependents();
        return;
    }
    load_tables(sK, sPad, pad);
    __syncthreads();
    pk::pdl_wait(tokens, tok_off, key_off, keys);
    if (R == 0) return;
    // all chunks, in tiles of one block, grid-strided
    const int64_t g_end = __ldcg(key_off + R);
    const uint32_t nblocks = gridDim.x - dw.desc_blocks;
    for (int64_t tile = (int64_t)(blockIdx.x - dw.desc_blocks) * kDigestBlock; tile < g_end;
         tile += (int64_t)nblocks * kDigestBlock) {
        const int64_t g = tile + threadIdx.x;
        const int64_t g0 = g - (threadIdx.x & 31);
        if (g0 >= g_end) break;  // whole warp past the end (uniform per warp)
        const uint32_t r = pk::lane_request_guess(key_off, R, g0, g_end, g);
        if (g < g_end) digest_chunk<F>(tokens, tok_off, key_off, r, g, C, sK, sPad, ring, keys, one);
        __syncwarp();
    }
    pk::pdl_launch_dependents();
}

// ---------------------------------------------------------------------------
// Chain: k_i = SHA-256(k_{i-1} || d || c_i), serial in i for each request.
//
// Every 32 requests (one per lane, a "group") are served by a pair of warps:
//   rounds warp:   holds the state; runs the 64 rounds of block 1
//                  (k_{i-1} || d) and of block 2 (c_i || padding)
//   schedule warp: writes K_t + W_t for both blocks to shared memory:
//                  block 2's schedule depends on c_i only and is made one
//                  step ahead; block 1's depends on k_{i-1} and is made as
//                  soon as k_{i-1} is published.
// Two layouts (kPairs):
//   1  one pair per CTA (2 warps) for batches with at most one group per SM:
//      the two warps run on different SM sub-partitions, so that one chain
//      step costs about the rounds alone; block 1's schedule is published in
//      three 16-word slices.  Named barriers (count 64, producer arrives,
//      consumer syncs): 1, 2, 3 block-1 slices t = 16..31, 32..47, 48..63;
//      4 block-2 schedule; 5 k_i published.
//   4  four pairs per CTA (8 warps), pair p = rounds warp p and schedule warp
//      p + 4, which share a sub-partition, one CTA per SM: with several
//      groups per SM, 2-warp CTAs put two rounds warps on one sub-partition
//      (51 instead of 30 cycles per round, measured) while schedule warps
//      share another; paired on one sub-partition, the schedule fills the
//      issue slots the rounds warp's dependency chain leaves idle.  Block 1's
//      schedule is published in two slices, t = 16..31 and 32..63 (the rounds
//      warp waits for the burst of block-1 schedule work after each k_{i-1},
//      so the smaller first slice lets its rounds 16..31 overlap the rest:
//      small-block key derivation 654 -> 641 us; three slices: 646).  The
//      first slice's barrier also marks block 2 of the step ready (written
//      before it), which keeps the pairs within the 16 named barriers.  Named
//      barriers of pair p: 1 + 3p block-1 slice 1 and block 2; 2 + 3p block-1
//      slice 2; 3 + 3p k_i published.
// Per pair both warps run the same number of steps (the lanes' maximum), so
// every phase of every barrier gets exactly one arrive and one sync; the
// schedule warp signals the block-2 barrier for step i only after it has
// passed the k barrier of step i-1 (so after the rounds warp has synced the
// block-2 barrier of step i-1), and the block-1 barriers of step i only after
// the k barrier of step i-1 (after the rounds warp's block-1 syncs of step
// i-1): it never arrives twice on a barrier the rounds warp has not yet
// synced.  Block 2's buffer for step i + 1 is written after the k barrier of
// step i - 1, when the rounds warp has finished the block 2 that last used
// it.  Lanes past their own request's last chunk keep computing (masked) so
// that the warps stay aligned.
// ---------------------------------------------------------------------------
constexpr int kChainLanes = 32;

__device__ __forceinline__ void bar_sync(int id) { asm volatile("bar.sync %0, 64;" ::"r"(id) : "memory"); }
__device__ __forceinline__ void bar_arrive(int id) { asm volatile("bar.arrive %0, 64;" ::"r"(id) : "memory"); }

// K+W words pass between the two warps four to a 16-byte vector ([t / 4][lane]): one shared-memory
// instruction per four words on either side.
struct ChainSmem {
    uint4 kw1[16][kChainLanes];     // block-1 K+W, t = 16..63 used
    uint4 kw2[2][16][kChainLanes];  // block-2 K+W, double-buffered by step parity
    uint4 kpub[2][kChainLanes];     // k_{i-1} for the schedule warp
};

// 16 schedule words t = 16q .. 16q+15 of the ring w (in place), K_t + W_t -> out[t / 4][lane]
// (F: round form of pk_sha256.cuh, `one` its run-time 1)
template <int F>
__device__ __forceinline__ void schedule16(uint32_t w[16], uint4 (*out)[kChainLanes], int q, uint32_t lane,
                                           uint32_t one) {
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        pk::sched_word<F>(w, j, one);
        o[j & 3] = pk::add2<F>(pk::kSha256K[16 * q + j], w[j], one);
        if ((j & 3) == 3) out[4 * q + (j >> 2)][lane] = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

// rounds t = 16q .. 16q+15 with K+W from shared memory
// (the 16 words are read into registers before the first round: a lone warp
// runs 64 rounds in 2018 instead of 2241 cycles when no round waits on its
// shared-memory read)
template <int F>
__device__ __forceinline__ void rounds16_kw(uint32_t v[8], const uint4 (*kw)[kChainLanes], int q, uint32_t lane,
                                            uint32_t one) {
    uint32_t a = v[0], b = v[1], c = v[2], d = v[3], e = v[4], f = v[5], g = v[6], h = v[7];
    uint32_t x[16];
#pragma unroll
    for (int m = 0; m < 4; ++m) {
        const uint4 y = kw[4 * q + m][lane];
        x[4 * m] = y.x;
        x[4 * m + 1] = y.y;
        x[4 * m + 2] = y.z;
        x[4 * m + 3] = y.w;
    }
#pragma unroll
    for (int j = 0; j < 16; ++j) pk::round_kw<F>(a, b, c, d, e, f, g, h, x[j], one);
    v[0] = a; v[1] = b; v[2] = c; v[3] = d; v[4] = e; v[5] = f; v[6] = g; v[7] = h;
}

// At most 64 registers (no spills): uncapped, the compiler took 81 and a small-block step whose
// lookup-and-store launch overlaps the chain's tail ran 910 -> 955 us.  `groups` = ceil(R / 32); with
// kPairs = 4, CTA c serves groups [c * groups / gridDim.x, (c + 1) * groups / gridDim.x), at most four.
// FS1, FS2: the forms (pk_sha256.cuh) of the schedule warp's additions for block 1 and block 2, `one` their
// run-time 1 (with one pair per CTA the two blocks share one loop and FS1).  The rounds warp keeps the
// compiler's form: its dependency chain sets the step time, and a multiply-add's longer latency there made
// the four-pair chain slower (small-block key derivation 674 -> 718 us with every addition on the FMA pipe).
// With four pairs each sub-partition runs a rounds warp and a schedule warp, whose two blocks differ:
// block 1's schedule (k_{i-1} || d) can start only when k_{i-1} is published, and the rounds warp waits for
// it after its 16th round, so it keeps the short-latency form; block 2's (c_i || padding) is made a step
// ahead, off the critical path, and its additions go to the FMA pipe, where they do not compete with the
// rounds warp's logic.  Small-block key derivation, measured: 683.7 us with both blocks in one loop and all
// schedule additions on the FMA pipe; 674.8 with all on the ALU; 661.9 with the blocks in two loops, all on
// the ALU; 655.8 as here.  Moving the small sigmas' shifts or rotations to the FMA pipe as well (mul.hi /
// mad.lo by 2^(32-n): 4 and 6 cycles per warp instruction there) lost on either block (666-707 us): the
// rounds warp's own multiply-adds queue behind them.  Block 2's first 16 words (K_t + W_t, set by
// block2_head) and step 0's whole block 2, made before the loop, take FS1: 668 -> 654 us against FS2.
template <int kPairs, int FS1, int FS2>
__global__ void __launch_bounds__(2 * kChainLanes * kPairs, kPairs == 1 ? 15 : 4)
k_chain(const int64_t *key_off, const uint32_t *desc_idx,
        const uint8_t *digests, uint32_t R, uint32_t D, uint8_t *keys, uint32_t groups, uint32_t one) {
    extern __shared__ __align__(16) uint8_t chain_smem[];
    pk::pdl_wait(key_off, desc_idx, digests, keys);  // successor released at the last step (see k_chunk_digest)
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t pair = kPairs == 1 ? 0u : warp & (kPairs - 1);
    const bool sched = kPairs == 1 ? warp == 1 : warp >= (uint32_t)kPairs;
    ChainSmem &sm = reinterpret_cast<ChainSmem *>(chain_smem)[pair];
    uint32_t group = blockIdx.x;
    bool active = true;
    if (kPairs > 1) {
        const uint32_t g0 = (uint32_t)((uint64_t)blockIdx.x * groups / gridDim.x);
        const uint32_t g1 = (uint32_t)((uint64_t)(blockIdx.x + 1) * groups / gridDim.x);
        group = g0 + pair;
        active = group < g1;
    }
    // named barriers of this pair (compile-time ids with one pair per CTA)
    const int bar_s1 = kPairs == 1 ? 1 : 1 + 3 * (int)pair;  // block-1 schedule (first slice)
    const int bar_s1b = kPairs == 1 ? 2 : 2 + 3 * (int)pair;  // block-1 schedule (second slice)
    const int bar_b2 = kPairs == 1 ? 4 : -1;                  // block-2 schedule (four pairs: with bar_s1)
    const int bar_k = kPairs == 1 ? 5 : 3 + 3 * (int)pair;   // k_i published
    const uint32_t r = group * kChainLanes + lane;
    int64_t a = 0, n = 0;
    uint32_t di = 0;
    if (active && r < R) {
        a = key_off[r];
        n = key_off[r + 1] - a;
        di = desc_idx[r];
        if (n < 0 || di >= D) n = 0;
    }
    int64_t nmax = n;  // identical in both warps of the pair: they cover the same 32 requests
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const int64_t x = __shfl_xor_sync(0xffffffffu, nmax, o);
        nmax = x > nmax ? x : nmax;
    }
    if (nmax == 0) {  // uniform over the pair
        pk::pdl_launch_dependents();
        if (kPairs > 1) __syncthreads();
        return;
    }

    uint32_t dw[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    if (n > 0) {
        const uint4 *dq = reinterpret_cast<const uint4 *>(digests + 32ull * di);
        const uint4 d_lo = __ldcg(dq), d_hi = __ldcg(dq + 1);
        dw[0] = pk::bswap32(d_lo.x); dw[1] = pk::bswap32(d_lo.y); dw[2] = pk::bswap32(d_lo.z);
        dw[3] = pk::bswap32(d_lo.w); dw[4] = pk::bswap32(d_hi.x); dw[5] = pk::bswap32(d_hi.y);
        dw[6] = pk::bswap32(d_hi.z); dw[7] = pk::bswap32(d_hi.w);
    }
    uint4 *kq = reinterpret_cast<uint4 *>(keys + 32ull * a);

    if (sched) {  // ---------------- schedule warp ----------------
        // With one pair per CTA, one loop runs one copy of the 16-word schedule body for all six slices
        // of a step (block-1 slices 1-3 of step i, then block-2 slices 1-3 of step i+1): the rounds warp
        // on the next sub-partition slows down with the amount of distinct code this warp runs (per chain
        // step, measured: 2206 ns with four unrolled copies, 2085 ns with one; 1950 ns with no schedule
        // work at all).  With four pairs the two blocks have a loop each, in their own forms (FS1, FS2).
        // block 2 of step i: W = c_i (8 words) || 0x80000000, 0 x 6, 768; words 0..15 stored as K + W
        auto block2_head = [&](int64_t i, int buf, uint32_t w[16]) {
            if (i < n) {
                const uint4 lo = kq[2 * i], hi = kq[2 * i + 1];
                w[0] = pk::bswap32(lo.x); w[1] = pk::bswap32(lo.y); w[2] = pk::bswap32(lo.z); w[3] = pk::bswap32(lo.w);
                w[4] = pk::bswap32(hi.x); w[5] = pk::bswap32(hi.y); w[6] = pk::bswap32(hi.z); w[7] = pk::bswap32(hi.w);
            } else {
#pragma unroll
                for (int j = 0; j < 8; ++j) w[j] = 0;
            }
            w[8] = 0x80000000u;
#pragma unroll
            for (int j = 9; j < 15; ++j) w[j] = 0;
            w[15] = 96u * 8u;
#pragma unroll
            for (int m = 0; m < 4; ++m)
                sm.kw2[buf][m][lane] = make_uint4(
                    pk::add2<FS1>(pk::kSha256K[4 * m], w[4 * m], one), pk::add2<FS1>(pk::kSha256K[4 * m + 1], w[4 * m + 1], one),
                    pk::add2<FS1>(pk::kSha256K[4 * m + 2], w[4 * m + 2], one),
                    pk::add2<FS1>(pk::kSha256K[4 * m + 3], w[4 * m + 3], one));
        };
        {
            uint32_t w[16];
            block2_head(0, 0, w);
#pragma unroll 1
            for (int q = 1; q < 4; ++q) schedule16<FS1>(w, sm.kw2[0], q, lane, one);
        }
        if (kPairs == 1) bar_arrive(bar_b2);
#pragma unroll 1
        for (int64_t i = 0; i < nmax; ++i) {
            if (i + 1 == nmax) pk::pdl_launch_dependents();
            uint32_t w[16];
            if (i == 0) {
#pragma unroll
                for (int j = 0; j < 8; ++j) w[j] = 0;  // k_{-1} = 0^32
            } else {
                bar_sync(bar_k);  // k_{i-1} published; the rounds warp has finished step i-1
#pragma unroll
                for (int m = 0; m < 2; ++m) {
                    const uint4 y = sm.kpub[m][lane];
                    w[4 * m] = y.x;
                    w[4 * m + 1] = y.y;
                    w[4 * m + 2] = y.z;
                    w[4 * m + 3] = y.w;
                }
                if (kPairs == 1) bar_arrive(bar_b2);  // block-2 schedule of step i (made in the previous iteration)
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) w[8 + j] = dw[j];
            const int buf = (int)((i + 1) & 1);
            if (kPairs == 1) {
                const int slices = i + 1 < nmax ? 6 : 3;
#pragma unroll 1
                for (int sl = 1; sl <= slices; ++sl) {
                    if (sl == 4) block2_head(i + 1, buf, w);
                    schedule16<FS1>(w, sl <= 3 ? sm.kw1 : sm.kw2[buf], sl <= 3 ? sl : sl - 3, lane, one);
                    // constant barrier ids (a run-time id reserves all 16 named barriers)
                    if (sl == 1) bar_arrive(1);
                    else if (sl == 2) bar_arrive(2);
                    else if (sl == 3) bar_arrive(3);
                }
            } else {
                schedule16<FS1>(w, sm.kw1, 1, lane, one);
                bar_arrive(bar_s1);  // also: block 2 of step i ready
#pragma unroll 1
                for (int sl = 2; sl <= 3; ++sl) schedule16<FS1>(w, sm.kw1, sl, lane, one);
                bar_arrive(bar_s1b);
                if (i + 1 < nmax) {
                    block2_head(i + 1, buf, w);
#pragma unroll 1
                    for (int sl = 1; sl <= 3; ++sl) schedule16<FS2>(w, sm.kw2[buf], sl, lane, one);
                }
            }
        }
        __syncthreads();  // stay resident until the rounds warp has consumed every phase
        return;
    }

    // ---------------- rounds warp ----------------
    uint32_t p[8] = {0, 0, 0, 0, 0, 0, 0, 0};  // k_{-1} = 0^32
    uint32_t kd[8];                            // K_t + d_{t-8}, t = 8..15
#pragma unroll
    for (int j = 0; j < 8; ++j) kd[j] = pk::kSha256K[8 + j] + dw[j];
#pragma unroll 1
    for (int64_t i = 0; i < nmax; ++i) {
        if (i + 1 == nmax) pk::pdl_launch_dependents();
        uint32_t v[8] = {PK_IV0, PK_IV1, PK_IV2, PK_IV3, PK_IV4, PK_IV5, PK_IV6, PK_IV7};
        {   // block 1, rounds 0..15: W = k_{i-1} || d
            uint32_t a_ = v[0], b_ = v[1], c_ = v[2], d_ = v[3], e_ = v[4], f_ = v[5], g_ = v[6], h_ = v[7];
#pragma unroll
            for (int j = 0; j < 8; ++j) pk::round_kw(a_, b_, c_, d_, e_, f_, g_, h_, pk::kSha256K[j] + p[j]);
#pragma unroll
            for (int j = 0; j < 8; ++j) pk::round_kw(a_, b_, c_, d_, e_, f_, g_, h_, kd[j]);
            v[0] = a_; v[1] = b_; v[2] = c_; v[3] = d_; v[4] = e_; v[5] = f_; v[6] = g_; v[7] = h_;
        }
        if (kPairs == 1) {
            bar_sync(1);
            rounds16_kw<pk::kAddsPlain>(v, sm.kw1, 1, lane, one);
            bar_sync(2);
            rounds16_kw<pk::kAddsPlain>(v, sm.kw1, 2, lane, one);
            bar_sync(3);
            rounds16_kw<pk::kAddsPlain>(v, sm.kw1, 3, lane, one);
        } else {
            bar_sync(bar_s1);
            rounds16_kw<pk::kAddsPlain>(v, sm.kw1, 1, lane, one);
            bar_sync(bar_s1b);
            rounds16_kw<pk::kAddsPlain>(v, sm.kw1, 2, lane, one);
            rounds16_kw<pk::kAddsPlain>(v, sm.kw1, 3, lane, one);
        }
        uint32_t st[8] = {PK_IV0 + v[0], PK_IV1 + v[1], PK_IV2 + v[2], PK_IV3 + v[3],
                          PK_IV4 + v[4], PK_IV5 + v[5], PK_IV6 + v[6], PK_IV7 + v[7]};
        if (kPairs == 1) bar_sync(bar_b2);  // block-2 schedule of step i
        const uint4 (*kw2)[kChainLanes] = sm.kw2[i & 1];
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = st[j];
#pragma unroll 1
        for (int q = 0; q < 4; ++q) rounds16_kw<pk::kAddsPlain>(v, kw2, q, lane, one);
#pragma unroll
        for (int j = 0; j < 8; ++j) p[j] = st[j] + v[j];
        if (i < n) store_digest(keys + 32ull * (a + i), p);
        if (i + 1 < nmax) {
#pragma unroll
            for (int m = 0; m < 2; ++m) sm.kpub[m][lane] = make_uint4(p[4 * m], p[4 * m + 1], p[4 * m + 2], p[4 * m + 3]);
            bar_arrive(bar_k);
        }
    }
    __syncthreads();
}

unsigned grid_for(uint64_t n, unsigned block) { return (unsigned)((n + block - 1) / block); }

// Shared memory of the four-pair chain CTA: its four ChainSmem (100 KiB), padded past half of an SM's
// shared memory so that no SM holds two of these CTAs (the launch becomes resident while the chunk digests
// drain, and would otherwise stack CTAs on the SMs that free up first).
constexpr size_t kChainPackedSmem = 116 * 1024;
static_assert(kChainPackedSmem >= 4 * sizeof(ChainSmem), "four pairs fit");

// Raise the four-pair chain CTA's shared-memory limit once per device.
cudaError_t chain_packed_attr() {
    static std::mutex mu;
    static bool done[256] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 256) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!done[dev]) {
        e = cudaFuncSetAttribute(k_chain<4, pk::kAddsPlain, pk::kAddsFma>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kChainPackedSmem);
        if (e != cudaSuccess) return e;
        done[dev] = true;
    }
    return cudaSuccess;
}

}  // namespace

cudaError_t pk_launch_digest_descriptors(const uint8_t *enc, uint64_t enc_bytes, const int64_t *enc_off,
                                         uint32_t D, uint8_t *digests, int32_t *status, cudaStream_t s) {
    if (D == 0) return cudaSuccess;
    const cudaError_t e =
        pk_launch(k_digest_descriptors, grid_for(D, kDescWarps), 32 * kDescWarps, s, enc, enc_bytes, enc_off, D,
                  digests, status);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t pk_launch_derive(const pk_ctx *ctx, const int32_t *tokens, uint64_t n_tokens,
                             const int64_t *tok_off, uint32_t R, const uint32_t *desc_idx,
                             const uint8_t *digests, uint32_t D, int64_t *key_off, uint8_t *keys,
                             uint64_t key_capacity, int32_t *status, cudaStream_t s) {
    return pk_launch_derive_enc(ctx, tokens, n_tokens, tok_off, R, desc_idx, nullptr, 0, nullptr, D,
                                const_cast<uint8_t *>(digests), key_off, keys, key_capacity, status, s);
}

cudaError_t pk_launch_derive_enc(const pk_ctx *ctx, const int32_t *tokens, uint64_t n_tokens,
                                 const int64_t *tok_off, uint32_t R, const uint32_t *desc_idx, const uint8_t *enc,
                                 uint64_t enc_bytes, const int64_t *enc_off, uint32_t D, uint8_t *digests,
                                 int64_t *key_off, uint8_t *keys, uint64_t key_capacity, int32_t *status,
                                 cudaStream_t s) {
    static_assert(kDigestBlock / 32 * kDescStage <= (int)sizeof(uint32_t) * kStages * kDigestBlock * 16,
                  "descriptor staging fits in the token ring");
    const uint32_t C = ctx->chunk_tokens;
    cudaError_t e = pk_launch(k_chunk_offsets, 1, kScanThreads, s, tok_off, R, n_tokens, C, desc_idx, D, key_capacity,
                              key_off, status);
    if (e != cudaSuccess) return e;
    DescWork dw = {enc, enc_bytes, enc_off, D, digests, status, 0};
    if (enc_off) dw.desc_blocks = grid_for(D, kDigestBlock / 32);
    PadKW pad;
    for (int t = 0; t < 64; ++t) pad.kw[t] = ctx->pad_kw[t];
    const bool chunks = R > 0 && key_capacity > 0;
    const uint32_t one = 1u;
    if (!chunks) {
        if (dw.desc_blocks)
            e = pk_launch(k_chunk_digest<pk::kAddsPlain>, dw.desc_blocks, kDigestBlock, s, tokens, tok_off,
                          (const int64_t *)key_off, 0u, C, pad, keys, dw, one);
        return e != cudaSuccess ? e : cudaGetLastError();
    }
    // The multiply-add round form pays once at least kFmaWarps warps of chunks share each SM
    // sub-partition (measured 10-13% per compression at 4 warps; slower for a lone warp).  The chunk
    // count is at most key_capacity; with an unknown SM count the compiler's form is kept.
    const uint64_t warps = (key_capacity + 31) / 32;
    const bool fma = ctx->sm_count > 0 && warps >= (uint64_t)kFmaWarps * 4u * ctx->sm_count;
    const unsigned grid = grid_for(key_capacity, kDigestBlock) + dw.desc_blocks;
    e = fma ? pk_launch(k_chunk_digest<pk::kAddsFma>, grid, kDigestBlock, s, tokens, tok_off, (const int64_t *)key_off,
                        R, C, pad, keys, dw, one)
            : pk_launch(k_chunk_digest<pk::kAddsPlain>, grid, kDigestBlock, s, tokens, tok_off,
                        (const int64_t *)key_off, R, C, pad, keys, dw, one);
    if (e != cudaSuccess) return e;
    // Chains: one pair per CTA while the groups of 32 requests fit one per SM; four pairs per CTA (one CTA
    // per SM, each pair on its own sub-partition) for more groups.
    const uint32_t groups = grid_for(R, kChainLanes);
    if (ctx->sm_count == 0 || groups <= ctx->sm_count) {
        e = pk_launch_smem(k_chain<1, pk::kAddsPlain, pk::kAddsPlain>, groups, 2 * kChainLanes, sizeof(ChainSmem), s,
                           (const int64_t *)key_off, desc_idx, (const uint8_t *)digests, R, D, keys, groups, one);
    } else {
        e = chain_packed_attr();
        const uint32_t grid = groups <= 4 * ctx->sm_count ? ctx->sm_count : grid_for(groups, 4);
        if (e == cudaSuccess)
            e = pk_launch_smem(k_chain<4, pk::kAddsPlain, pk::kAddsFma>, grid, 8 * kChainLanes, kChainPackedSmem, s,
                               (const int64_t *)key_off, desc_idx, (const uint8_t *)digests, R, D, keys, groups, one);
    }
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}
