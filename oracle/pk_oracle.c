/*
 * pk_oracle.c -- CPU oracle for provenance-bound KV-cache key derivation.
 *
 * TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only tests/, __graft_entry__.smoke()
 * and the cpu_baseline / reference leg of bench.py may load this library.  It
 * shares no code, header, table or constant with the CUDA path: the SHA-256
 * constants below are derived at start-up from their FIPS 180-4 definitions
 * instead of being typed in.
 *
 * Plain, slow and obviously correct by design: every message is padded into a
 * freshly allocated buffer exactly as FIPS 180-4 section 5.1.1 describes and
 * then hashed block by block (section 6.2.2), with no precomputation, fusion
 * or reordering.
 *
 * What it computes (Eq. 3 of the paper, Key(x,c) = f(x, H(enc(...))), with
 * H = SHA-256 and the connector key function f instantiated as a chained
 * per-chunk digest):
 *   c_i = SHA-256(LE-int32 bytes of tokens[iC, (i+1)C))          chunk digest
 *   k_i = SHA-256(k_{i-1} || d || c_i),  k_{-1} = 32 zero bytes   chained key
 * for the n_r = floor(T_r / C) full chunks of each request r; a trailing
 * partial chunk gets no key (Sec. 4.4: prefixes below one chunk never collide).
 *
 * Pins: SHA-256 against hashlib (OpenSSL) and the FIPS 180-2 Appendix B
 * example digests; chunk serialisation against the same published digests
 * re-expressed as int32 tokens; the chain against the contract invariants
 * (Eqs. 1, 2 and 4) by brute force.  The byte order of the chain message
 * (k_{i-1} before d before c_i) and the zero seed are stated conventions that
 * the paper leaves open: parity unpinned by the paper for those two choices.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ---------------------------------------------------------------------- */
/* Constants from their definitions (FIPS 180-4 sections 4.2.2 and 5.3.3). */
/* ---------------------------------------------------------------------- */

static uint32_t K[64];  /* first 32 bits of the fractional parts of the cube roots of the first 64 primes */
static uint32_t H0[8];  /* first 32 bits of the fractional parts of the square roots of the first 8 primes */
static int constants_ready = 0;

static int is_prime(unsigned n) {
    if (n < 2) return 0;
    for (unsigned q = 2; q * q <= n; ++q)
        if (n % q == 0) return 0;
    return 1;
}

/* floor(cbrt(p) * 2^32) by bisection on x^3 <= p * 2^96, exact in 128-bit integers. */
static uint64_t floor_cbrt_scaled(unsigned p) {
    unsigned __int128 target = (unsigned __int128)p << 96;
    uint64_t lo = 0, hi = (uint64_t)1 << 40;  /* cbrt(311) < 8, so the answer is below 2^35 */
    while (hi - lo > 1) {
        uint64_t mid = lo + (hi - lo) / 2;
        unsigned __int128 m = mid;
        if (m * m * m <= target) lo = mid; else hi = mid;
    }
    return lo;
}

/* floor(sqrt(p) * 2^32) by bisection on x^2 <= p * 2^64. */
static uint64_t floor_sqrt_scaled(unsigned p) {
    unsigned __int128 target = (unsigned __int128)p << 64;
    uint64_t lo = 0, hi = (uint64_t)1 << 40;
    while (hi - lo > 1) {
        uint64_t mid = lo + (hi - lo) / 2;
        unsigned __int128 m = mid;
        if (m * m <= target) lo = mid; else hi = mid;
    }
    return lo;
}

static void init_constants(void) {
    if (constants_ready) return;
    unsigned found = 0;
    for (unsigned n = 2; found < 64; ++n) {
        if (!is_prime(n)) continue;
        K[found] = (uint32_t)floor_cbrt_scaled(n);      /* keeps the low 32 bits = fractional part */
        if (found < 8) H0[found] = (uint32_t)floor_sqrt_scaled(n);
        ++found;
    }
    constants_ready = 1;
}

/* ---------------------------------------------------------------------- */
/* SHA-256, FIPS 180-4 section 6.2                                          */
/* ---------------------------------------------------------------------- */

static uint32_t rotr(uint32_t x, unsigned n) { return (x >> n) | (x << (32u - n)); }
static uint32_t ch(uint32_t x, uint32_t y, uint32_t z) { return (x & y) ^ (~x & z); }
static uint32_t maj(uint32_t x, uint32_t y, uint32_t z) { return (x & y) ^ (x & z) ^ (y & z); }
static uint32_t big_sigma0(uint32_t x) { return rotr(x, 2) ^ rotr(x, 13) ^ rotr(x, 22); }
static uint32_t big_sigma1(uint32_t x) { return rotr(x, 6) ^ rotr(x, 11) ^ rotr(x, 25); }
static uint32_t small_sigma0(uint32_t x) { return rotr(x, 7) ^ rotr(x, 18) ^ (x >> 3); }
static uint32_t small_sigma1(uint32_t x) { return rotr(x, 17) ^ rotr(x, 19) ^ (x >> 10); }

void oracle_sha256(const uint8_t *msg, uint64_t len, uint8_t out[32]) {
    init_constants();

    /* 5.1.1: append the bit 1, then k zero bits with len*8 + 1 + k = 448 mod 512,
     * then the 64-bit big-endian bit length. */
    uint64_t padded = ((len + 8) / 64 + 1) * 64;
    uint8_t *m = (uint8_t *)calloc((size_t)padded, 1);
    if (len) memcpy(m, msg, (size_t)len);
    m[len] = 0x80;
    uint64_t bits = len * 8u;
    for (int b = 0; b < 8; ++b) m[padded - 1 - b] = (uint8_t)(bits >> (8 * b));

    uint32_t Hs[8];
    for (int j = 0; j < 8; ++j) Hs[j] = H0[j];

    for (uint64_t blk = 0; blk < padded / 64; ++blk) {
        const uint8_t *M = m + 64 * blk;
        uint32_t W[64];
        /* 6.2.2 step 1: message schedule; words are read big-endian (section 3.1). */
        for (int t = 0; t < 16; ++t)
            W[t] = ((uint32_t)M[4 * t] << 24) | ((uint32_t)M[4 * t + 1] << 16) |
                   ((uint32_t)M[4 * t + 2] << 8) | (uint32_t)M[4 * t + 3];
        for (int t = 16; t < 64; ++t)
            W[t] = small_sigma1(W[t - 2]) + W[t - 7] + small_sigma0(W[t - 15]) + W[t - 16];
        /* step 2: working variables */
        uint32_t a = Hs[0], b = Hs[1], c = Hs[2], d = Hs[3];
        uint32_t e = Hs[4], f = Hs[5], g = Hs[6], h = Hs[7];
        /* step 3: 64 rounds */
        for (int t = 0; t < 64; ++t) {
            uint32_t T1 = h + big_sigma1(e) + ch(e, f, g) + K[t] + W[t];
            uint32_t T2 = big_sigma0(a) + maj(a, b, c);
            h = g; g = f; f = e; e = d + T1;
            d = c; c = b; b = a; a = T1 + T2;
        }
        /* step 4: intermediate hash value */
        Hs[0] += a; Hs[1] += b; Hs[2] += c; Hs[3] += d;
        Hs[4] += e; Hs[5] += f; Hs[6] += g; Hs[7] += h;
    }
    free(m);
    /* the digest is H_0 .. H_7, each word big-endian */
    for (int j = 0; j < 8; ++j) {
        out[4 * j + 0] = (uint8_t)(Hs[j] >> 24);
        out[4 * j + 1] = (uint8_t)(Hs[j] >> 16);
        out[4 * j + 2] = (uint8_t)(Hs[j] >> 8);
        out[4 * j + 3] = (uint8_t)(Hs[j]);
    }
}

/* ---------------------------------------------------------------------- */
/* Key derivation                                                           */
/* ---------------------------------------------------------------------- */

/* Serialise n int32 tokens as little-endian bytes, one byte at a time. */
static void tokens_to_le_bytes(const int32_t *tok, uint64_t n, uint8_t *out) {
    for (uint64_t j = 0; j < n; ++j) {
        uint32_t u = (uint32_t)tok[j];
        out[4 * j + 0] = (uint8_t)(u);
        out[4 * j + 1] = (uint8_t)(u >> 8);
        out[4 * j + 2] = (uint8_t)(u >> 16);
        out[4 * j + 3] = (uint8_t)(u >> 24);
    }
}

/* c = SHA-256(LE bytes of C tokens) */
void oracle_chunk_digest(const int32_t *tok, uint32_t C, uint8_t c_out[32]) {
    uint8_t *bytes = (uint8_t *)malloc((size_t)C * 4 + 1);
    tokens_to_le_bytes(tok, C, bytes);
    oracle_sha256(bytes, (uint64_t)C * 4, c_out);
    free(bytes);
}

/* k = SHA-256(prev || d || c) over the 96-byte concatenation */
void oracle_chain_step(const uint8_t prev[32], const uint8_t d[32], const uint8_t c[32],
                       uint8_t k_out[32]) {
    uint8_t msg[96];
    memcpy(msg, prev, 32);
    memcpy(msg + 32, d, 32);
    memcpy(msg + 64, c, 32);
    oracle_sha256(msg, 96, k_out);
}

/* All keys of one request of T tokens under descriptor digest d.
 * Writes floor(T/C) keys of 32 bytes and returns that count. */
uint64_t oracle_request_keys(const int32_t *tok, uint64_t T, uint32_t C, const uint8_t d[32],
                             uint8_t *keys_out) {
    uint64_t n = T / C;
    uint8_t prev[32];
    memset(prev, 0, 32);                      /* k_{-1} = 32 zero bytes */
    for (uint64_t i = 0; i < n; ++i) {
        uint8_t c[32];
        oracle_chunk_digest(tok + i * C, C, c);
        oracle_chain_step(prev, d, c, keys_out + 32 * i);
        memcpy(prev, keys_out + 32 * i, 32);
    }
    return n;
}

/* Batch form.  tok_off has R+1 entries; request r is tokens[tok_off[r], tok_off[r+1]).
 * key_off_out gets R+1 entries: key_off[r+1] = key_off[r] + floor(T_r / C).
 * digests holds D descriptor digests of 32 bytes; request r uses digests[desc_idx[r]].
 * Returns the number of keys, or -1 on a bad argument. */
int64_t oracle_derive_keys(const int32_t *tokens, const int64_t *tok_off, uint32_t R, uint32_t C,
                           const uint32_t *desc_idx, const uint8_t *digests, uint32_t D,
                           int64_t *key_off_out, uint8_t *keys_out) {
    if (C == 0) return -1;
    init_constants();                        /* once, before the parallel loop */
    key_off_out[0] = 0;
    for (uint32_t r = 0; r < R; ++r) {
        if (tok_off[r + 1] < tok_off[r] || desc_idx[r] >= D) return -1;
        key_off_out[r + 1] = key_off_out[r] + (tok_off[r + 1] - tok_off[r]) / C;
    }
    /* Requests are independent; the loop over them is the only parallelism. */
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < (int64_t)R; ++r) {
        oracle_request_keys(tokens + tok_off[r], (uint64_t)(tok_off[r + 1] - tok_off[r]), C,
                            digests + 32 * (uint64_t)desc_idx[r], keys_out + 32 * key_off_out[r]);
    }
    return key_off_out[R];
}

int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* Exposed so that a test can check the derived constants' internal
 * consistency; the digests themselves are pinned against hashlib. */
void oracle_constants(uint32_t k_out[64], uint32_t h_out[8]) {
    init_constants();
    memcpy(k_out, K, sizeof K);
    memcpy(h_out, H0, sizeof H0);
}
