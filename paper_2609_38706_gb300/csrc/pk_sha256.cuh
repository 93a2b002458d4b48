// pk_sha256.cuh -- SHA-256 compression for the CUDA path (device) and the
// library's host-side descriptor digest.
//
// FIPS 180-4: section 6.2.2 (compression), 4.2.2 (round constants), 5.3.3
// (initial hash value), 5.1.1 (padding).  SHA-256 is the collision-resistant
// hash H of the paper's canonical realization (Sec. 5.2, Eq. 3) and the
// content / chain digest of the key function.
//
// The 64 rounds are written out with literal round constants so that they
// become instruction immediates; message words are passed by value so that a
// caller passing constants (padding blocks, fixed message tails) has its
// message schedule folded at compile time.  Rotations are funnel shifts on
// the device.
#pragma once
#include <stdint.h>

#if defined(__CUDACC__)
#define PK_HD __host__ __device__ __forceinline__
#else
#define PK_HD static inline
#endif

namespace pk {

// Initial hash value H(0) (FIPS 180-4 section 5.3.3).
#define PK_IV0 0x6a09e667u
#define PK_IV1 0xbb67ae85u
#define PK_IV2 0x3c6ef372u
#define PK_IV3 0xa54ff53au
#define PK_IV4 0x510e527fu
#define PK_IV5 0x9b05688cu
#define PK_IV6 0x1f83d9abu
#define PK_IV7 0x5be0cd19u

PK_HD uint32_t rotr(uint32_t x, int n) {
#if defined(__CUDA_ARCH__)
    return __funnelshift_r(x, x, n);
#else
    return (x >> n) | (x << (32 - n));
#endif
}

// Big-endian word <-> little-endian memory word.
PK_HD uint32_t bswap32(uint32_t x) {
#if defined(__CUDA_ARCH__)
    return __byte_perm(x, 0u, 0x0123u);
#else
    return __builtin_bswap32(x);
#endif
}

PK_HD uint32_t big_s0(uint32_t a) { return rotr(a, 2) ^ rotr(a, 13) ^ rotr(a, 22); }
PK_HD uint32_t big_s1(uint32_t e) { return rotr(e, 6) ^ rotr(e, 11) ^ rotr(e, 25); }
PK_HD uint32_t small_s0(uint32_t w) { return rotr(w, 7) ^ rotr(w, 18) ^ (w >> 3); }
PK_HD uint32_t small_s1(uint32_t w) { return rotr(w, 17) ^ rotr(w, 19) ^ (w >> 10); }
PK_HD uint32_t ch(uint32_t e, uint32_t f, uint32_t g) { return (e & f) ^ (~e & g); }
PK_HD uint32_t maj(uint32_t a, uint32_t b, uint32_t c) { return (a & b) | (c & (a | b)); }

// One round: T1 = h + S1(e) + Ch(e,f,g) + K_t + W_t; T2 = S0(a) + Maj(a,b,c);
// d += T1; h = T1 + T2.  The caller rotates the variable names each round.
#define PK_RND(a, b, c, d, e, f, g, h, k, w)                                  \
    {                                                                          \
        uint32_t t1_ = (h) + big_s1(e) + ch(e, f, g) + (k) + (w);             \
        uint32_t t2_ = big_s0(a) + maj(a, b, c);                              \
        (d) += t1_;                                                            \
        (h) = t1_ + t2_;                                                       \
    }

// Message schedule in a 16-word ring: W_t = s1(W_{t-2}) + W_{t-7} + s0(W_{t-15}) + W_{t-16}.
#define PK_SCHED(wt, wt15, wt7, wt2) ((wt) += small_s1(wt2) + (wt7) + small_s0(wt15))

// state <- state + compress(state, W[0..15])
PK_HD void compress(uint32_t st[8],
                    uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3,
                    uint32_t w4, uint32_t w5, uint32_t w6, uint32_t w7,
                    uint32_t w8, uint32_t w9, uint32_t w10, uint32_t w11,
                    uint32_t w12, uint32_t w13, uint32_t w14, uint32_t w15) {
    uint32_t a = st[0], b = st[1], c = st[2], d = st[3];
    uint32_t e = st[4], f = st[5], g = st[6], h = st[7];
    PK_RND(a, b, c, d, e, f, g, h, 0x428a2f98u, w0);
    PK_RND(h, a, b, c, d, e, f, g, 0x71374491u, w1);
    PK_RND(g, h, a, b, c, d, e, f, 0xb5c0fbcfu, w2);
    PK_RND(f, g, h, a, b, c, d, e, 0xe9b5dba5u, w3);
    PK_RND(e, f, g, h, a, b, c, d, 0x3956c25bu, w4);
    PK_RND(d, e, f, g, h, a, b, c, 0x59f111f1u, w5);
    PK_RND(c, d, e, f, g, h, a, b, 0x923f82a4u, w6);
    PK_RND(b, c, d, e, f, g, h, a, 0xab1c5ed5u, w7);
    PK_RND(a, b, c, d, e, f, g, h, 0xd807aa98u, w8);
    PK_RND(h, a, b, c, d, e, f, g, 0x12835b01u, w9);
    PK_RND(g, h, a, b, c, d, e, f, 0x243185beu, w10);
    PK_RND(f, g, h, a, b, c, d, e, 0x550c7dc3u, w11);
    PK_RND(e, f, g, h, a, b, c, d, 0x72be5d74u, w12);
    PK_RND(d, e, f, g, h, a, b, c, 0x80deb1feu, w13);
    PK_RND(c, d, e, f, g, h, a, b, 0x9bdc06a7u, w14);
    PK_RND(b, c, d, e, f, g, h, a, 0xc19bf174u, w15);
    PK_RND(a, b, c, d, e, f, g, h, 0xe49b69c1u, PK_SCHED(w0, w1, w9, w14));
    PK_RND(h, a, b, c, d, e, f, g, 0xefbe4786u, PK_SCHED(w1, w2, w10, w15));
    PK_RND(g, h, a, b, c, d, e, f, 0x0fc19dc6u, PK_SCHED(w2, w3, w11, w0));
    PK_RND(f, g, h, a, b, c, d, e, 0x240ca1ccu, PK_SCHED(w3, w4, w12, w1));
    PK_RND(e, f, g, h, a, b, c, d, 0x2de92c6fu, PK_SCHED(w4, w5, w13, w2));
    PK_RND(d, e, f, g, h, a, b, c, 0x4a7484aau, PK_SCHED(w5, w6, w14, w3));
    PK_RND(c, d, e, f, g, h, a, b, 0x5cb0a9dcu, PK_SCHED(w6, w7, w15, w4));
    PK_RND(b, c, d, e, f, g, h, a, 0x76f988dau, PK_SCHED(w7, w8, w0, w5));
    PK_RND(a, b, c, d, e, f, g, h, 0x983e5152u, PK_SCHED(w8, w9, w1, w6));
    PK_RND(h, a, b, c, d, e, f, g, 0xa831c66du, PK_SCHED(w9, w10, w2, w7));
    PK_RND(g, h, a, b, c, d, e, f, 0xb00327c8u, PK_SCHED(w10, w11, w3, w8));
    PK_RND(f, g, h, a, b, c, d, e, 0xbf597fc7u, PK_SCHED(w11, w12, w4, w9));
    PK_RND(e, f, g, h, a, b, c, d, 0xc6e00bf3u, PK_SCHED(w12, w13, w5, w10));
    PK_RND(d, e, f, g, h, a, b, c, 0xd5a79147u, PK_SCHED(w13, w14, w6, w11));
    PK_RND(c, d, e, f, g, h, a, b, 0x06ca6351u, PK_SCHED(w14, w15, w7, w12));
    PK_RND(b, c, d, e, f, g, h, a, 0x14292967u, PK_SCHED(w15, w0, w8, w13));
    PK_RND(a, b, c, d, e, f, g, h, 0x27b70a85u, PK_SCHED(w0, w1, w9, w14));
    PK_RND(h, a, b, c, d, e, f, g, 0x2e1b2138u, PK_SCHED(w1, w2, w10, w15));
    PK_RND(g, h, a, b, c, d, e, f, 0x4d2c6dfcu, PK_SCHED(w2, w3, w11, w0));
    PK_RND(f, g, h, a, b, c, d, e, 0x53380d13u, PK_SCHED(w3, w4, w12, w1));
    PK_RND(e, f, g, h, a, b, c, d, 0x650a7354u, PK_SCHED(w4, w5, w13, w2));
    PK_RND(d, e, f, g, h, a, b, c, 0x766a0abbu, PK_SCHED(w5, w6, w14, w3));
    PK_RND(c, d, e, f, g, h, a, b, 0x81c2c92eu, PK_SCHED(w6, w7, w15, w4));
    PK_RND(b, c, d, e, f, g, h, a, 0x92722c85u, PK_SCHED(w7, w8, w0, w5));
    PK_RND(a, b, c, d, e, f, g, h, 0xa2bfe8a1u, PK_SCHED(w8, w9, w1, w6));
    PK_RND(h, a, b, c, d, e, f, g, 0xa81a664bu, PK_SCHED(w9, w10, w2, w7));
    PK_RND(g, h, a, b, c, d, e, f, 0xc24b8b70u, PK_SCHED(w10, w11, w3, w8));
    PK_RND(f, g, h, a, b, c, d, e, 0xc76c51a3u, PK_SCHED(w11, w12, w4, w9));
    PK_RND(e, f, g, h, a, b, c, d, 0xd192e819u, PK_SCHED(w12, w13, w5, w10));
    PK_RND(d, e, f, g, h, a, b, c, 0xd6990624u, PK_SCHED(w13, w14, w6, w11));
    PK_RND(c, d, e, f, g, h, a, b, 0xf40e3585u, PK_SCHED(w14, w15, w7, w12));
    PK_RND(b, c, d, e, f, g, h, a, 0x106aa070u, PK_SCHED(w15, w0, w8, w13));
    PK_RND(a, b, c, d, e, f, g, h, 0x19a4c116u, PK_SCHED(w0, w1, w9, w14));
    PK_RND(h, a, b, c, d, e, f, g, 0x1e376c08u, PK_SCHED(w1, w2, w10, w15));
    PK_RND(g, h, a, b, c, d, e, f, 0x2748774cu, PK_SCHED(w2, w3, w11, w0));
    PK_RND(f, g, h, a, b, c, d, e, 0x34b0bcb5u, PK_SCHED(w3, w4, w12, w1));
    PK_RND(e, f, g, h, a, b, c, d, 0x391c0cb3u, PK_SCHED(w4, w5, w13, w2));
    PK_RND(d, e, f, g, h, a, b, c, 0x4ed8aa4au, PK_SCHED(w5, w6, w14, w3));
    PK_RND(c, d, e, f, g, h, a, b, 0x5b9cca4fu, PK_SCHED(w6, w7, w15, w4));
    PK_RND(b, c, d, e, f, g, h, a, 0x682e6ff3u, PK_SCHED(w7, w8, w0, w5));
    PK_RND(a, b, c, d, e, f, g, h, 0x748f82eeu, PK_SCHED(w8, w9, w1, w6));
    PK_RND(h, a, b, c, d, e, f, g, 0x78a5636fu, PK_SCHED(w9, w10, w2, w7));
    PK_RND(g, h, a, b, c, d, e, f, 0x84c87814u, PK_SCHED(w10, w11, w3, w8));
    PK_RND(f, g, h, a, b, c, d, e, 0x8cc70208u, PK_SCHED(w11, w12, w4, w9));
    PK_RND(e, f, g, h, a, b, c, d, 0x90befffau, PK_SCHED(w12, w13, w5, w10));
    PK_RND(d, e, f, g, h, a, b, c, 0xa4506cebu, PK_SCHED(w13, w14, w6, w11));
    PK_RND(c, d, e, f, g, h, a, b, 0xbef9a3f7u, PK_SCHED(w14, w15, w7, w12));
    PK_RND(b, c, d, e, f, g, h, a, 0xc67178f2u, PK_SCHED(w15, w0, w8, w13));
    st[0] += a; st[1] += b; st[2] += c; st[3] += d;
    st[4] += e; st[5] += f; st[6] += g; st[7] += h;
}

PK_HD void compress16(uint32_t st[8], const uint32_t w[16]) {
    compress(st, w[0], w[1], w[2], w[3], w[4], w[5], w[6], w[7],
             w[8], w[9], w[10], w[11], w[12], w[13], w[14], w[15]);
}

PK_HD void init_state(uint32_t st[8]) {
    st[0] = PK_IV0; st[1] = PK_IV1; st[2] = PK_IV2; st[3] = PK_IV3;
    st[4] = PK_IV4; st[5] = PK_IV5; st[6] = PK_IV6; st[7] = PK_IV7;
}

}  // namespace pk

namespace pk {

// SHA-256 of an arbitrary byte string (FIPS 180-4 5.1.1 padding assembled on
// the fly, bytes loaded one at a time).  Used for short messages only: the
// descriptor encodings.
PK_HD void sha256_bytes(const uint8_t *p, uint64_t len, uint8_t out[32]) {
    uint32_t st[8];
    init_state(st);
    const uint64_t nblocks = (len + 8) / 64 + 1;
    const uint64_t bits = len * 8u;
    for (uint64_t blk = 0; blk < nblocks; ++blk) {
        uint32_t w[16];
        for (int t = 0; t < 16; ++t) {
            uint32_t v = 0;
            for (int q = 0; q < 4; ++q) {
                const uint64_t idx = blk * 64 + 4 * t + q;
                const uint32_t byte = idx < len ? p[idx] : (idx == len ? 0x80u : 0u);
                v = (v << 8) | byte;
            }
            w[t] = v;
        }
        if (blk == nblocks - 1) {
            w[14] = (uint32_t)(bits >> 32);
            w[15] = (uint32_t)bits;
        }
        compress16(st, w);
    }
    for (int j = 0; j < 8; ++j) {
        out[4 * j + 0] = (uint8_t)(st[j] >> 24);
        out[4 * j + 1] = (uint8_t)(st[j] >> 16);
        out[4 * j + 2] = (uint8_t)(st[j] >> 8);
        out[4 * j + 3] = (uint8_t)(st[j]);
    }
}

}  // namespace pk

#if defined(__CUDACC__)
namespace pk {

// Device-side compression with the 64 rounds written as a 16-round body that
// is executed four times (the message schedule ring has period 16, and the
// working-variable rotation period 8 divides 16, so one body serves all four
// quarters).  Keeping the code a quarter of the fully unrolled size keeps a
// loop of several compressions resident in the instruction cache; the round
// constants are read from a shared-memory copy (sK, 64 words) that each
// kernel makes at its start.
//
// Pipes.  Every rotation, shift and 3-input logic operation of SHA-256 issues
// on the SM's ALU pipe, one warp instruction per 2 cycles per sub-partition,
// and so do the 3-input integer adds the compiler emits for most additions
// (measured on GB300: SHF, LOP3 and IADD3 each 2.0 cycles per warp
// instruction).  An integer multiply-add issues on the FMA pipe, at the same
// rate and alongside the ALU (an SHF/IMAD pair: 2.1 cycles).  The two round
// forms differ only in where the additions go, never in the value computed:
//   kAddsPlain  the compiler's choice (ALU-bound at 25 cycles per round when
//               the sub-partition is saturated, 29.8 for a lone warp);
//   kAddsFma    every addition as x * one + y on the FMA pipe (`one` is a
//               run-time 1 the compiler cannot fold): 22.2 cycles per round
//               and 10-13% faster compressions once 4 or more warps share a
//               sub-partition, but 33.4 cycles for a lone warp (the
//               multiply-add's longer latency sits on the critical path).
enum { kAddsPlain = 0, kAddsFma = 1 };

// x * one + c, kept as a multiply-add (one == 1 at run time).
__device__ __forceinline__ uint32_t mad1(uint32_t x, uint32_t one, uint32_t c) {
    uint32_t r;
    asm("mad.lo.u32 %0, %1, %2, %3;" : "=r"(r) : "r"(x), "r"(one), "r"(c));
    return r;
}

template <int F = kAddsPlain>
__device__ __forceinline__ uint32_t add2(uint32_t x, uint32_t y, uint32_t one) {
    if (F == kAddsFma) return mad1(x, one, y);
    return x + y;
}

template <int F = kAddsPlain>
__device__ __forceinline__ void round_kw(uint32_t &a, uint32_t &b, uint32_t &c, uint32_t &d, uint32_t &e,
                                         uint32_t &f, uint32_t &g, uint32_t &h, uint32_t kw, uint32_t one = 1u) {
    if (F == kAddsFma) {
        const uint32_t t1 = mad1(big_s1(e), one, mad1(ch(e, f, g), one, mad1(h, one, kw)));
        const uint32_t t2 = mad1(big_s0(a), one, maj(a, b, c));
        h = g; g = f; f = e; e = mad1(d, one, t1); d = c; c = b; b = a; a = mad1(t1, one, t2);
    } else {
        const uint32_t t1 = h + big_s1(e) + ch(e, f, g) + kw;
        const uint32_t t2 = big_s0(a) + maj(a, b, c);
        h = g; g = f; f = e; e = d + t1; d = c; c = b; b = a; a = t1 + t2;
    }
}

// W_t = s1(W_{t-2}) + W_{t-7} + s0(W_{t-15}) + W_{t-16} in the 16-word ring w, slot j.
template <int F = kAddsPlain>
__device__ __forceinline__ uint32_t sched_word(uint32_t w[16], int j, uint32_t one) {
    if (F == kAddsFma)
        w[j] = mad1(small_s1(w[(j + 14) & 15]), one,
                    mad1(small_s0(w[(j + 1) & 15]), one, mad1(w[(j + 9) & 15], one, w[j])));
    else
        w[j] += small_s1(w[(j + 14) & 15]) + w[(j + 9) & 15] + small_s0(w[(j + 1) & 15]);
    return w[j];
}

template <bool SCHED, int F = kAddsPlain>
__device__ __forceinline__ void rounds16(uint32_t v[8], uint32_t w[16], const uint32_t *__restrict__ k16,
                                         uint32_t one = 1u) {
    uint32_t a = v[0], b = v[1], c = v[2], d = v[3], e = v[4], f = v[5], g = v[6], h = v[7];
    uint32_t k[16];  // read before the first round, so that no round waits on shared memory
#pragma unroll
    for (int j = 0; j < 16; ++j) k[j] = k16[j];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        if (SCHED) sched_word<F>(w, j, one);
        round_kw<F>(a, b, c, d, e, f, g, h, add2<F>(k[j], w[j], one), one);
    }
    v[0] = a; v[1] = b; v[2] = c; v[3] = d; v[4] = e; v[5] = f; v[6] = g; v[7] = h;
}

// st <- st + compress(st, w); w is overwritten by the schedule.
template <int F = kAddsPlain>
__device__ __forceinline__ void compress_rolled(uint32_t st[8], uint32_t w[16], const uint32_t *__restrict__ sK,
                                                uint32_t one = 1u) {
    uint32_t v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = st[j];
    rounds16<false, F>(v, w, sK, one);
#pragma unroll 1
    for (int q = 1; q < 4; ++q) rounds16<true, F>(v, w, sK + 16 * q, one);
#pragma unroll
    for (int j = 0; j < 8; ++j) st[j] = add2<F>(st[j], v[j], one);
}

// st <- st + compress(st, W) for a message whose whole schedule is known in
// advance: kw[t] = K_t + W_t for t = 0..63 (rounds only).
template <int F = kAddsPlain>
__device__ __forceinline__ void compress_kw(uint32_t st[8], const uint32_t *__restrict__ kw, uint32_t one = 1u) {
    uint32_t a = st[0], b = st[1], c = st[2], d = st[3], e = st[4], f = st[5], g = st[6], h = st[7];
#pragma unroll 1
    for (int q = 0; q < 4; ++q) {
        uint32_t x[16];  // read before the first round, as in rounds16
#pragma unroll
        for (int j = 0; j < 16; ++j) x[j] = kw[16 * q + j];
#pragma unroll
        for (int j = 0; j < 16; ++j) round_kw<F>(a, b, c, d, e, f, g, h, x[j], one);
    }
    st[0] = add2<F>(st[0], a, one); st[1] = add2<F>(st[1], b, one); st[2] = add2<F>(st[2], c, one);
    st[3] = add2<F>(st[3], d, one); st[4] = add2<F>(st[4], e, one); st[5] = add2<F>(st[5], f, one);
    st[6] = add2<F>(st[6], g, one); st[7] = add2<F>(st[7], h, one);
}

}  // namespace pk
#endif

namespace pk {

// FIPS 180-4 round constants K_0..K_63 (section 4.2.2), as data for the
// shared-memory copy used by the device compressions.
#define PK_K_TABLE                                                                                   \
    0x428a2f98u, 0x71374491u, 0xb5c0fbcfu, 0xe9b5dba5u, 0x3956c25bu, 0x59f111f1u, 0x923f82a4u,       \
        0xab1c5ed5u, 0xd807aa98u, 0x12835b01u, 0x243185beu, 0x550c7dc3u, 0x72be5d74u, 0x80deb1feu,   \
        0x9bdc06a7u, 0xc19bf174u, 0xe49b69c1u, 0xefbe4786u, 0x0fc19dc6u, 0x240ca1ccu, 0x2de92c6fu,   \
        0x4a7484aau, 0x5cb0a9dcu, 0x76f988dau, 0x983e5152u, 0xa831c66du, 0xb00327c8u, 0xbf597fc7u,   \
        0xc6e00bf3u, 0xd5a79147u, 0x06ca6351u, 0x14292967u, 0x27b70a85u, 0x2e1b2138u, 0x4d2c6dfcu,   \
        0x53380d13u, 0x650a7354u, 0x766a0abbu, 0x81c2c92eu, 0x92722c85u, 0xa2bfe8a1u, 0xa81a664bu,   \
        0xc24b8b70u, 0xc76c51a3u, 0xd192e819u, 0xd6990624u, 0xf40e3585u, 0x106aa070u, 0x19a4c116u,   \
        0x1e376c08u, 0x2748774cu, 0x34b0bcb5u, 0x391c0cb3u, 0x4ed8aa4au, 0x5b9cca4fu, 0x682e6ff3u,   \
        0x748f82eeu, 0x78a5636fu, 0x84c87814u, 0x8cc70208u, 0x90befffau, 0xa4506cebu, 0xbef9a3f7u,   \
        0xc67178f2u

#if defined(__CUDACC__)
// Device copy of the round constants (one per translation unit), the source of
// the shared-memory tables the compressions read.
static __constant__ uint32_t kSha256K[64] = {PK_K_TABLE};
#endif

// Schedule-plus-constant table of a message block known on the host:
// kw[t] = K_t + W_t (used for the constant final padding block of a chunk).
PK_HD void kw_table(const uint32_t m[16], uint32_t kw[64]) {
    const uint32_t K[64] = {PK_K_TABLE};
    uint32_t W[64];
    for (int t = 0; t < 16; ++t) W[t] = m[t];
    for (int t = 16; t < 64; ++t) W[t] = small_s1(W[t - 2]) + W[t - 7] + small_s0(W[t - 15]) + W[t - 16];
    for (int t = 0; t < 64; ++t) kw[t] = K[t] + W[t];
}

}  // namespace pk
