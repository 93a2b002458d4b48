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
// Output bytes dominate the traffic (the row width against 16 key bytes read
// per row), so the kernel is built to write at HBM speed: a persistent grid,
// each CTA holding two tiles of 256 rows in shared memory, laid out exactly
// as in the output (256 * width bytes, a multiple of 16) and filled once with
// the prefix and zeros.  Per tile only the 22 characters of each row change:
// every thread encodes its key into its row, then one thread hands the whole
// tile to the TMA engine as a single bulk store (cp.async.bulk, shared to
// global).  The two tiles alternate, so encoding the next tile overlaps the
// store of the previous one, and each thread's next key is loaded a tile
// ahead.
#include <cuda_runtime.h>

#include <mutex>

#include "pk_device.cuh"
#include "pk_internal.h"

namespace {

constexpr uint32_t kRows = 256;  // rows per tile; one thread per row
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

// Bulk copy of `bytes` (a multiple of 16) from shared to global memory,
// tracked in this thread's bulk group.
__device__ __forceinline__ void bulk_store(void *gdst, const void *ssrc, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;"
                 :
                 : "l"(gdst), "r"((uint32_t)__cvta_generic_to_shared(ssrc)), "r"(bytes)
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// At most one bulk group of this thread still reading shared memory.
__device__ __forceinline__ void bulk_wait_read_1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
// Every bulk group of this thread complete.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// Shared-memory writes of this thread visible to the TMA engine (async proxy).
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void encode_row(const uint4 &k, uint8_t *c) {
    // The 16 bytes as a 128-bit big-endian integer (hi, lo); character q is
    // bits [6q, 6q + 6) counted from the most significant bit.
    const uint64_t hi = ((uint64_t)bswap32(k.x) << 32) | bswap32(k.y);
    const uint64_t lo = ((uint64_t)bswap32(k.z) << 32) | bswap32(k.w);
#pragma unroll
    for (uint32_t q = 0; q < kChars; ++q) {
        const uint32_t s = 6 * q;  // <= 126
        const uint64_t top = s == 0 ? hi : s < 64 ? (hi << s) | (lo >> (64 - s)) : lo << (s - 64);
        c[q] = b64_char((uint32_t)(top >> 58));
    }
}

__global__ void __launch_bounds__(kRows) k_key_strings(const uint8_t *keys, uint64_t n, KeyStrArgs a, uint8_t *out) {
    extern __shared__ __align__(128) uint8_t sm[];  // two tiles of kRows * width bytes
    const uint32_t t = threadIdx.x;
    const uint32_t tile_bytes = kRows * a.width;
    // Both tiles: zeros, then the prefix at the start of every row.
    uint4 *sm4 = reinterpret_cast<uint4 *>(sm);
    for (uint32_t i = t; i < 2 * tile_bytes / 16; i += kRows) sm4[i] = make_uint4(0, 0, 0, 0);
    __syncthreads();
    for (uint32_t j = 0; j < a.plen; ++j) {
        sm[t * a.width + j] = a.prefix[j];
        sm[tile_bytes + t * a.width + j] = a.prefix[j];
    }
    pk::pdl_wait(keys, out);
    const uint64_t n_tiles = (n + kRows - 1) / kRows;
    uint64_t tile = blockIdx.x;
    uint4 k = make_uint4(0, 0, 0, 0);
    if (tile * kRows + t < n) k = __ldcg(reinterpret_cast<const uint4 *>(keys + 32 * (tile * kRows + t)));
    for (uint32_t it = 0; tile < n_tiles; tile += gridDim.x, ++it) {
        uint8_t *buf = sm + (it & 1) * tile_bytes;
        const uint64_t row0 = tile * kRows;
        const uint32_t rows = (uint32_t)min((uint64_t)kRows, n - row0);
        const uint64_t next = row0 + (uint64_t)gridDim.x * kRows + t;  // this thread's key of the next tile
        uint4 k_next = make_uint4(0, 0, 0, 0);
        if (next < n) k_next = __ldcg(reinterpret_cast<const uint4 *>(keys + 32 * next));
        if (t == 0) bulk_wait_read_1();  // the store that last used `buf` has read it
        __syncthreads();
        if (t < rows) encode_row(k, buf + t * a.width + a.plen);
        fence_proxy_async_smem();
        __syncthreads();
        const uint32_t bytes = rows * a.width;
        const uint32_t b16 = bytes & ~15u;
        uint8_t *dst = out + row0 * a.width;  // 16-byte aligned: 256 * width is a multiple of 16
        if (t == 0 && b16) bulk_store(dst, buf, b16);
        for (uint32_t j = b16 + t; j < bytes; j += kRows) dst[j] = buf[j];  // the last tile's final bytes
        k = k_next;
    }
    pk::pdl_launch_dependents();
    if (t == 0) bulk_wait_all();  // shared memory stays allocated until the TMA engine has read it
}

}  // namespace

// Resident CTAs of k_key_strings for a row width (SMs x CTAs per SM), computed
// once per device and width; the first call also raises the kernel's dynamic
// shared-memory limit to the largest width's two tiles.
static cudaError_t keystr_resident(int dev, uint32_t width, uint64_t *out) {
    static std::mutex mu;
    static uint32_t sms[256] = {};
    static uint16_t per_sm[256][PK_KEY_STRING_MAX_WIDTH + 1] = {};
    if (dev < 0 || dev >= 256 || width > PK_KEY_STRING_MAX_WIDTH) return cudaErrorInvalidValue;
    std::lock_guard<std::mutex> lock(mu);
    if (!sms[dev]) {
        int n = 0;
        cudaError_t e = cudaFuncSetAttribute(k_key_strings, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)(2 * kRows * PK_KEY_STRING_MAX_WIDTH));
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
        sms[dev] = (uint32_t)n;
    }
    if (!per_sm[dev][width]) {
        int b = 0;
        const cudaError_t e =
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, k_key_strings, kRows, 2ull * kRows * width);
        if (e != cudaSuccess) return e;
        per_sm[dev][width] = (uint16_t)(b < 1 ? 1 : b);
    }
    *out = (uint64_t)sms[dev] * per_sm[dev][width];
    return cudaSuccess;
}

cudaError_t pk_launch_key_strings(const uint8_t *keys, uint64_t n, const uint8_t *prefix, uint32_t plen,
                                  uint32_t width, uint8_t *out, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    KeyStrArgs a;
    a.plen = plen;
    a.width = width;
    for (uint32_t j = 0; j < PK_KEY_STRING_MAX_WIDTH; ++j) a.prefix[j] = j < plen ? prefix[j] : 0;
    const size_t smem = 2ull * kRows * width;  // <= 128 KiB
    int dev = 0;
    uint64_t resident = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = keystr_resident(dev, width, &resident);
    if (e != cudaSuccess) return e;
    const uint64_t tiles = (n + kRows - 1) / kRows;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(tiles < resident ? tiles : resident));
    cfg.blockDim = dim3(kRows);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, k_key_strings, keys, n, a, out);
    return e != cudaSuccess ? e : cudaGetLastError();
}
