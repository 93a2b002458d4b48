// pk_keystr.cu -- connector key strings of a key batch (Sec. 5.3, connector
// integration).  A connector whose wire format is a fixed-width text field
// carries the 128-bit digest as twenty-two base64 characters: the standard
// alphabet of RFC 4648, Sec. 4, with the two "=" of padding dropped (16 bytes
// give 21 full 6-bit groups and 2 leftover bits, the last character's low
// four bits zero).  Row i of the output is
//     prefix || base64(first 16 bytes of k_i) || zero bytes up to the row width
// where the prefix (the connector's fixed fields and the model tag) is the
// same for every row.
//
// The rows of 256 keys form one contiguous tile of the output (256 * width is
// a multiple of 16), written as coalesced 16-byte stores: each thread first
// encodes the 22 characters of one key into shared memory, then the block
// assembles the tile 16 bytes per thread from the prefix, the characters and
// zeros.  Output bytes dominate the traffic (width against 16 key bytes read
// per row), so the kernel is bound by HBM writes.
#include <cuda_runtime.h>

#include "pk_device.cuh"
#include "pk_internal.h"

namespace {

constexpr uint32_t kRows = 256;  // keys (rows) per block; also threads per block
constexpr uint32_t kChars = PK_KEY_STRING_CHARS;

struct KeyStrArgs {
    uint32_t plen;   // prefix bytes
    uint32_t width;  // row width in bytes, plen + 22 <= width <= PK_KEY_STRING_MAX_WIDTH
    uint8_t prefix[PK_KEY_STRING_MAX_WIDTH];
};

__device__ __forceinline__ uint8_t b64_char(uint32_t v) {  // v < 64
    return (uint8_t)(v < 26 ? 'A' + v : v < 52 ? 'a' + (v - 26) : v < 62 ? '0' + (v - 52) : v == 62 ? '+' : '/');
}

__device__ __forceinline__ uint32_t bswap32(uint32_t x) { return __byte_perm(x, 0, 0x0123); }

__global__ void __launch_bounds__(kRows) k_key_strings(const uint8_t *keys, uint64_t n, KeyStrArgs a, uint8_t *out) {
    __shared__ uint8_t pre[PK_KEY_STRING_MAX_WIDTH];
    __shared__ uint8_t chars[kRows * kChars];
    pk::pdl_wait(keys, out);
    const uint32_t t = threadIdx.x;
    const uint64_t row0 = (uint64_t)blockIdx.x * kRows;
    const uint32_t rows = (uint32_t)min((uint64_t)kRows, n - row0);
    for (uint32_t j = t; j < a.plen; j += kRows) pre[j] = a.prefix[j];
    if (t < rows) {
        // The 16 bytes as a 128-bit big-endian integer (hi, lo); character q
        // is bits [6q, 6q + 6) counted from the most significant bit.
        const uint4 k = __ldcg(reinterpret_cast<const uint4 *>(keys + 32 * (row0 + t)));
        const uint64_t hi = ((uint64_t)bswap32(k.x) << 32) | bswap32(k.y);
        const uint64_t lo = ((uint64_t)bswap32(k.z) << 32) | bswap32(k.w);
        uint8_t *c = chars + t * kChars;
#pragma unroll
        for (uint32_t q = 0; q < kChars; ++q) {
            const uint32_t s = 6 * q;  // <= 126
            const uint64_t top = s == 0 ? hi : s < 64 ? (hi << s) | (lo >> (64 - s)) : lo << (s - 64);
            c[q] = b64_char((uint32_t)(top >> 58));
        }
    }
    __syncthreads();
    // Tile bytes [0, rows * width); unit u = bytes [16u, 16u + 16).
    const uint64_t bytes = (uint64_t)rows * a.width;
    uint8_t *dst = out + row0 * a.width;
    for (uint64_t u = t; 16 * u < bytes; u += kRows) {
        uint64_t o = 16 * u;
        uint32_t r = (uint32_t)(o / a.width), col = (uint32_t)(o - (uint64_t)r * a.width);
        uint32_t w[4] = {0, 0, 0, 0};
        const uint32_t nb = (uint32_t)min((uint64_t)16, bytes - o);
#pragma unroll
        for (uint32_t b = 0; b < 16; ++b) {
            if (b < nb) {
                const uint32_t v =
                    col < a.plen ? pre[col] : col < a.plen + kChars ? chars[r * kChars + col - a.plen] : 0u;
                w[b >> 2] |= v << (8 * (b & 3));
                if (++col == a.width) {
                    col = 0;
                    ++r;
                }
            }
        }
        if (nb == 16) {
            *reinterpret_cast<uint4 *>(dst + o) = make_uint4(w[0], w[1], w[2], w[3]);
        } else {  // the last bytes of the last tile
#pragma unroll
            for (uint32_t b = 0; b < 16; ++b)
                if (b < nb) dst[o + b] = (uint8_t)(w[b >> 2] >> (8 * (b & 3)));
        }
    }
    pk::pdl_launch_dependents();
}

}  // namespace

cudaError_t pk_launch_key_strings(const uint8_t *keys, uint64_t n, const uint8_t *prefix, uint32_t plen,
                                  uint32_t width, uint8_t *out, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    KeyStrArgs a;
    a.plen = plen;
    a.width = width;
    for (uint32_t j = 0; j < PK_KEY_STRING_MAX_WIDTH; ++j) a.prefix[j] = j < plen ? prefix[j] : 0;
    const cudaError_t e = pk_launch(k_key_strings, (unsigned)((n + kRows - 1) / kRows), kRows, s, keys, n, a, out);
    return e != cudaSuccess ? e : cudaGetLastError();
}
