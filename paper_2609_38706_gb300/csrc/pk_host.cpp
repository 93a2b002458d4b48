// pk_host.cpp -- host half of libpk: argument checks, descriptor
// canonicalisation and enc (Sec. 5.2-5.3), the host descriptor digest, and
// the C-ABI entry points that enqueue the kernels of pk_derive.cu / pk_table.cu.
#include <cuda_runtime_api.h>

#include <cstdlib>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "pk_internal.h"
#include "pk_sha256.cuh"

namespace {

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
// typed arrays must be naturally aligned (NULL passes; presence is checked separately)
bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

// Sec. 5.3, worker-level digest: bind the value the worker resolved, never a
// launch string such as "auto".  Resolved dtype names are compared ASCII
// case-insensitively and exact synonyms are folded to one spelling; distinct
// formats are never merged (a bare "fp8" stays "fp8").
int canonical_dtype(const pk_bytes &in, std::string *out) {
    if (in.len > PK_MAX_FIELD_BYTES) return PK_ERR_FIELD_TOO_LONG;
    if (in.len && !in.p) return PK_ERR_ARG;
    std::string s(reinterpret_cast<const char *>(in.p), in.len);
    for (char &c : s)
        if (c >= 'A' && c <= 'Z') c = (char)(c + 32);
    static const char *const kSyn[][2] = {
        {"bfloat16", "bf16"},          {"float16", "fp16"},         {"half", "fp16"},
        {"float32", "fp32"},           {"float", "fp32"},           {"float8_e4m3fn", "fp8_e4m3"},
        {"float8_e5m2", "fp8_e5m2"},
    };
    for (const auto &kv : kSyn)
        if (s == kv[0]) {
            s = kv[1];
            break;
        }
    if (s.empty() || s == "auto") return PK_ERR_UNRESOLVED;
    *out = s;
    return PK_OK;
}

int opaque(const pk_bytes &in, std::string *out) {
    if (in.len > PK_MAX_FIELD_BYTES) return PK_ERR_FIELD_TOO_LONG;
    if (in.len && !in.p) return PK_ERR_ARG;
    out->assign(reinterpret_cast<const char *>(in.p), in.len);
    return PK_OK;
}

void put_le32(std::string *dst, uint32_t v) {
    const char b[4] = {(char)(v & 0xff), (char)((v >> 8) & 0xff), (char)((v >> 16) & 0xff), (char)(v >> 24)};
    dst->append(b, 4);
}

// enc: LE32(number of fields) || for each field LE32(length) || bytes
// (Sec. 5.2, Eq. 3: injective, length-prefixed; appended fields per Prop. 1).
int encode(const pk_descriptor *d, std::string *enc) {
    if (!d) return PK_ERR_ARG;
    if (d->n_extra && !d->extra) return PK_ERR_ARG;
    std::string f[6];
    int rc;
    if ((rc = opaque(d->model_id, &f[0])) != PK_OK) return rc;
    if ((rc = canonical_dtype(d->weight_precision, &f[1])) != PK_OK) return rc;
    if ((rc = opaque(d->weight_version, &f[2])) != PK_OK) return rc;
    if ((rc = opaque(d->adapter_id, &f[3])) != PK_OK) return rc;
    if ((rc = canonical_dtype(d->kv_format, &f[4])) != PK_OK) return rc;
    if ((rc = opaque(d->salt, &f[5])) != PK_OK) return rc;
    enc->clear();
    put_le32(enc, 6u + d->n_extra);
    for (const auto &s : f) {
        put_le32(enc, (uint32_t)s.size());
        enc->append(s);
    }
    for (uint32_t j = 0; j < d->n_extra; ++j) {
        std::string x;
        if ((rc = opaque(d->extra[j], &x)) != PK_OK) return rc;
        put_le32(enc, (uint32_t)x.size());
        enc->append(x);
    }
    return PK_OK;
}

// Two-level variant (Sec. 2.2: request-level and worker-level provenance are
// bound through separate digests; Sec. 5.3: the worker-level digest is taken
// once over the resolved worker values, and the request-level binding is
// inert for a request with neither adapter nor salt).  Both halves use enc:
//   enc_w = LE32(4) || model id, weight precision, weight version, KV format
//   enc_q = LE32(2 + n_extra) || adapter id, salt, appended dimensions
int encode_worker(const pk_descriptor *d, std::string *enc) {
    if (!d) return PK_ERR_ARG;
    std::string f[4];
    int rc;
    if ((rc = opaque(d->model_id, &f[0])) != PK_OK) return rc;
    if ((rc = canonical_dtype(d->weight_precision, &f[1])) != PK_OK) return rc;
    if ((rc = opaque(d->weight_version, &f[2])) != PK_OK) return rc;
    if ((rc = canonical_dtype(d->kv_format, &f[3])) != PK_OK) return rc;
    enc->clear();
    put_le32(enc, 4u);
    for (const auto &s : f) {
        put_le32(enc, (uint32_t)s.size());
        enc->append(s);
    }
    return PK_OK;
}

int encode_request(const pk_descriptor *d, std::string *enc, bool *inert) {
    if (!d) return PK_ERR_ARG;
    if (d->n_extra && !d->extra) return PK_ERR_ARG;
    std::string f[2];
    int rc;
    if ((rc = opaque(d->adapter_id, &f[0])) != PK_OK) return rc;
    if ((rc = opaque(d->salt, &f[1])) != PK_OK) return rc;
    *inert = f[0].empty() && f[1].empty() && d->n_extra == 0;
    enc->clear();
    put_le32(enc, 2u + d->n_extra);
    for (const auto &s : f) {
        put_le32(enc, (uint32_t)s.size());
        enc->append(s);
    }
    for (uint32_t j = 0; j < d->n_extra; ++j) {
        std::string x;
        if ((rc = opaque(d->extra[j], &x)) != PK_OK) return rc;
        put_le32(enc, (uint32_t)x.size());
        enc->append(x);
    }
    return PK_OK;
}

// RFC 4648, Sec. 4, without padding: 16 bytes -> 22 characters.
void base64_16(const uint8_t *in, char *out) {
    static const char kAlphabet[] = "ABCDEFGHIJKLMNOPQRSTUVWXYZabcdefghijklmnopqrstuvwxyz0123456789+/";
    uint32_t acc = 0, bits = 0, o = 0;
    for (int i = 0; i < 16; ++i) {
        acc = (acc << 8) | in[i];
        bits += 8;
        while (bits >= 6) {
            bits -= 6;
            out[o++] = kAlphabet[(acc >> bits) & 63u];
        }
    }
    out[o] = kAlphabet[(acc << (6 - bits)) & 63u];  // 2 bits left, 4 zero bits appended
}

int cuda_rc(cudaError_t e) { return e == cudaSuccess ? PK_OK : PK_ERR_CUDA; }

}  // namespace

extern "C" {

size_t pk_table_bytes(uint32_t capacity_log2) {
    if (capacity_log2 < 1 || capacity_log2 > 31) return 0;
    return (size_t)PK_ENTRY_BYTES << capacity_log2;
}

int pk_init(pk_ctx **out, const pk_config *cfg, pk_stream stream) {
    if (!out) return PK_ERR_ARG;
    *out = nullptr;
    if (!cfg || cfg->chunk_tokens == 0 || !cfg->table_dev || !aligned16(cfg->table_dev)) return PK_ERR_ARG;
    const size_t need = pk_table_bytes(cfg->capacity_log2);
    if (need == 0 || cfg->table_bytes < need) return PK_ERR_CAPACITY;
    pk_ctx *c = new (std::nothrow) pk_ctx();
    if (!c) return PK_ERR_ARG;
    c->chunk_tokens = cfg->chunk_tokens;
    c->capacity_log2 = cfg->capacity_log2;
    c->capacity = 1ull << cfg->capacity_log2;
    c->max_probe = (cfg->max_probe == 0 || cfg->max_probe > c->capacity) ? (uint32_t)c->capacity : cfg->max_probe;
    c->table = static_cast<pk_entry *>(cfg->table_dev);
    c->epoch = 0;
    c->stamps = nullptr;
    c->sm_count = 0;
    {
        int dev = 0, sms = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && sms > 0)
            c->sm_count = (uint32_t)sms;
    }
    {   // final block of a 4C-byte message when 4C is a multiple of 64: 0x80, zeros, 64-bit bit length
        const uint64_t bits = (uint64_t)cfg->chunk_tokens * 32u;
        const uint32_t m[16] = {0x80000000u, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, (uint32_t)(bits >> 32),
                                (uint32_t)bits};
        pk::kw_table(m, c->pad_kw);
    }
    if (cudaMalloc(reinterpret_cast<void **>(&c->counter_dev), 256) != cudaSuccess) {
        delete c;
        return PK_ERR_CUDA;
    }
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(c->table, 0, need, s) != cudaSuccess ||
        cudaMemsetAsync(c->counter_dev, 0, 256, s) != cudaSuccess) {
        cudaFree(c->counter_dev);
        delete c;
        return PK_ERR_CUDA;
    }
    *out = c;
    return PK_OK;
}

int pk_destroy(pk_ctx *ctx) {
    if (!ctx) return PK_ERR_ARG;
    const cudaError_t e = cudaFree(ctx->counter_dev);
    delete ctx;
    return cuda_rc(e);
}

int pk_descriptor_encode(const pk_descriptor *desc, uint8_t *out, size_t cap, size_t *len) {
    std::string enc;
    const int rc = encode(desc, &enc);
    if (rc != PK_OK) return rc;
    if (len) *len = enc.size();
    if (enc.size() > cap || (!out && !enc.empty())) return PK_ERR_ARG;
    std::memcpy(out, enc.data(), enc.size());
    return PK_OK;
}

int pk_descriptors_encode(const pk_descriptor *descs, uint32_t D, uint8_t *out, size_t cap, int64_t *enc_off) {
    if (!enc_off || (D && !descs)) return PK_ERR_ARG;
    enc_off[0] = 0;
    size_t pos = 0;
    std::string enc;
    for (uint32_t j = 0; j < D; ++j) {
        const int rc = encode(descs + j, &enc);
        if (rc != PK_OK) return rc;
        if (pos + enc.size() > cap || !out) return PK_ERR_ARG;
        std::memcpy(out + pos, enc.data(), enc.size());
        pos += enc.size();
        enc_off[j + 1] = (int64_t)pos;
    }
    return PK_OK;
}

int pk_descriptor_digest(const pk_descriptor *desc, uint8_t out[32]) {
    if (!out) return PK_ERR_ARG;
    std::string enc;
    const int rc = encode(desc, &enc);
    if (rc != PK_OK) return rc;
    pk::sha256_bytes(reinterpret_cast<const uint8_t *>(enc.data()), enc.size(), out);
    return PK_OK;
}

int pk_worker_digest(const pk_descriptor *desc, uint8_t out[32]) {
    if (!out) return PK_ERR_ARG;
    std::string enc;
    const int rc = encode_worker(desc, &enc);
    if (rc != PK_OK) return rc;
    pk::sha256_bytes(reinterpret_cast<const uint8_t *>(enc.data()), enc.size(), out);
    return PK_OK;
}

int pk_request_digest(const uint8_t worker[32], const pk_descriptor *desc, uint8_t out[32]) {
    if (!worker || !out) return PK_ERR_ARG;
    std::string enc;
    bool inert = false;
    const int rc = encode_request(desc, &enc, &inert);
    if (rc != PK_OK) return rc;
    uint8_t msg[64];
    std::memcpy(msg, worker, 32);
    if (inert) {  // keys exactly as the worker-only chain
        std::memmove(out, msg, 32);
        return PK_OK;
    }
    pk::sha256_bytes(reinterpret_cast<const uint8_t *>(enc.data()), enc.size(), msg + 32);
    pk::sha256_bytes(msg, 64, out);
    return PK_OK;
}

int pk_request_digests(const uint8_t worker[32], const pk_descriptor *descs, uint32_t n, uint8_t *out) {
    if (n && (!descs || !out)) return PK_ERR_ARG;
    for (uint32_t j = 0; j < n; ++j) {
        const int rc = pk_request_digest(worker, descs + j, out + 32ull * j);
        if (rc != PK_OK) return rc;
    }
    return PK_OK;
}

int pk_digest_descriptors(pk_ctx *ctx, const uint8_t *enc_dev, uint64_t enc_bytes, const int64_t *enc_off_dev,
                          uint32_t D, uint8_t *digests_dev, int32_t *status_dev, pk_stream stream) {
    if (!ctx) return PK_ERR_ARG;
    if (D == 0) return PK_OK;
    if (!enc_off_dev || !digests_dev || (enc_bytes && !enc_dev) || !aligned(enc_off_dev, 8)) return PK_ERR_ARG;
    return cuda_rc(pk_launch_digest_descriptors(enc_dev, enc_bytes, enc_off_dev, D, digests_dev, status_dev,
                                                reinterpret_cast<cudaStream_t>(stream)));
}

int pk_derive_keys(pk_ctx *ctx, const int32_t *tokens_dev, uint64_t n_tokens, const int64_t *tok_off_dev,
                   uint32_t R, const uint32_t *desc_idx_dev, const uint8_t *digests_dev, uint32_t D,
                   int64_t *key_off_dev, uint8_t *keys_dev, uint64_t key_capacity, int32_t *status_dev,
                   pk_stream stream) {
    if (!ctx || !tok_off_dev || !key_off_dev) return PK_ERR_ARG;
    if (n_tokens && !tokens_dev) return PK_ERR_ARG;
    if (R && (!desc_idx_dev || !digests_dev || D == 0 || !aligned16(digests_dev))) return PK_ERR_ARG;
    if (key_capacity < n_tokens / ctx->chunk_tokens) return PK_ERR_ARG;
    if (key_capacity && (!keys_dev || !aligned16(keys_dev))) return PK_ERR_ARG;
    if (key_capacity > (uint64_t)0x7fffffff * 64) return PK_ERR_ARG;
    if (!aligned(tokens_dev, 4) || !aligned(tok_off_dev, 8) || !aligned(desc_idx_dev, 4) || !aligned(key_off_dev, 8))
        return PK_ERR_ARG;
    return cuda_rc(pk_launch_derive(ctx, tokens_dev, n_tokens, tok_off_dev, R, desc_idx_dev, digests_dev, D,
                                    key_off_dev, keys_dev, key_capacity, status_dev,
                                    reinterpret_cast<cudaStream_t>(stream)));
}

int pk_derive_keys_enc(pk_ctx *ctx, const int32_t *tokens_dev, uint64_t n_tokens, const int64_t *tok_off_dev,
                       uint32_t R, const uint32_t *desc_idx_dev, const uint8_t *enc_dev, uint64_t enc_bytes,
                       const int64_t *enc_off_dev, uint32_t D, uint8_t *digests_dev, int64_t *key_off_dev,
                       uint8_t *keys_dev, uint64_t key_capacity, int32_t *status_dev, pk_stream stream) {
    if (!ctx || !tok_off_dev || !key_off_dev) return PK_ERR_ARG;
    if (n_tokens && !tokens_dev) return PK_ERR_ARG;
    if (R && (!desc_idx_dev || D == 0)) return PK_ERR_ARG;
    if (D && (!enc_off_dev || !digests_dev || !aligned16(digests_dev) || !aligned(enc_off_dev, 8))) return PK_ERR_ARG;
    if (enc_bytes && !enc_dev) return PK_ERR_ARG;
    if (key_capacity < n_tokens / ctx->chunk_tokens) return PK_ERR_ARG;
    if (key_capacity && (!keys_dev || !aligned16(keys_dev))) return PK_ERR_ARG;
    if (key_capacity > (uint64_t)0x7fffffff * 64) return PK_ERR_ARG;
    if (!aligned(tokens_dev, 4) || !aligned(tok_off_dev, 8) || !aligned(desc_idx_dev, 4) || !aligned(key_off_dev, 8))
        return PK_ERR_ARG;
    return cuda_rc(pk_launch_derive_enc(ctx, tokens_dev, n_tokens, tok_off_dev, R, desc_idx_dev, enc_dev, enc_bytes,
                                        D ? enc_off_dev : nullptr, D, digests_dev, key_off_dev, keys_dev,
                                        key_capacity, status_dev, reinterpret_cast<cudaStream_t>(stream)));
}

int pk_lookup(pk_ctx *ctx, const uint8_t *keys_dev, const int64_t *key_off_dev, uint32_t R,
              uint64_t key_capacity, int32_t *hit_chunks_dev, uint32_t *slots_dev, int32_t *status_dev,
              pk_stream stream) {
    if (!ctx || !key_off_dev) return PK_ERR_ARG;
    if (R && !hit_chunks_dev) return PK_ERR_ARG;
    if (key_capacity && (!keys_dev || !aligned16(keys_dev) || !slots_dev)) return PK_ERR_ARG;
    if (key_capacity > (uint64_t)0x7fffffff * 256) return PK_ERR_ARG;
    if (!aligned(key_off_dev, 8) || !aligned(hit_chunks_dev, 4) || !aligned(slots_dev, 4)) return PK_ERR_ARG;
    return cuda_rc(pk_launch_lookup(ctx, keys_dev, key_off_dev, R, key_capacity, hit_chunks_dev, slots_dev,
                                    status_dev, reinterpret_cast<cudaStream_t>(stream)));
}

int pk_store(pk_ctx *ctx, const uint8_t *keys_dev, const uint32_t *slots_dev, uint64_t n,
             const int64_t *key_off_dev, const int32_t *hit_chunks_dev, uint32_t R, int32_t *result_dev,
             uint32_t *slot_out_dev, int32_t *status_dev, pk_stream stream) {
    if (!ctx) return PK_ERR_ARG;
    if ((key_off_dev == nullptr) != (hit_chunks_dev == nullptr)) return PK_ERR_ARG;
    if (n == 0) return PK_OK;
    if (!keys_dev || !aligned16(keys_dev) || !slots_dev || !result_dev || !slot_out_dev) return PK_ERR_ARG;
    if (n > (uint64_t)0x7fffffff * 256 || n >= 0xffffffffull) return PK_ERR_ARG;
    if (!aligned(slots_dev, 4) || !aligned(result_dev, 4) || !aligned(slot_out_dev, 4) || !aligned(key_off_dev, 8) ||
        !aligned(hit_chunks_dev, 4))
        return PK_ERR_ARG;
    const unsigned long long epoch = ++ctx->epoch;
    return cuda_rc(pk_launch_store(ctx, epoch, keys_dev, slots_dev, n, key_off_dev, hit_chunks_dev,
                                   key_off_dev ? R : 0, result_dev, slot_out_dev, status_dev,
                                   reinterpret_cast<cudaStream_t>(stream)));
}

int pk_lookup_store(pk_ctx *ctx, const uint8_t *keys_dev, const uint32_t *slots_new_dev, const int64_t *key_off_dev,
                    uint32_t R, uint64_t key_capacity, int32_t *hit_chunks_dev, uint32_t *slots_dev,
                    int32_t *result_dev, uint32_t *slot_out_dev, int32_t *status_dev, pk_stream stream) {
    if (!ctx || !key_off_dev) return PK_ERR_ARG;
    if (R && !hit_chunks_dev) return PK_ERR_ARG;
    if (key_capacity &&
        (!keys_dev || !aligned16(keys_dev) || !slots_new_dev || !slots_dev || !result_dev || !slot_out_dev))
        return PK_ERR_ARG;
    if (key_capacity > (uint64_t)0x7fffffff * 256 || key_capacity >= 0xffffffffull) return PK_ERR_ARG;
    if (!aligned(key_off_dev, 8) || !aligned(hit_chunks_dev, 4) || !aligned(slots_new_dev, 4) ||
        !aligned(slots_dev, 4) || !aligned(result_dev, 4) || !aligned(slot_out_dev, 4))
        return PK_ERR_ARG;
    const unsigned long long epoch = ++ctx->epoch;
    return cuda_rc(pk_launch_lookup_store(ctx, epoch, keys_dev, slots_new_dev, key_off_dev, R, key_capacity,
                                          hit_chunks_dev, slots_dev, result_dev, slot_out_dev, status_dev,
                                          reinterpret_cast<cudaStream_t>(stream)));
}

size_t pk_stamps_bytes(uint32_t capacity_log2) {
    if (capacity_log2 < 1 || capacity_log2 > 31) return 0;
    return (size_t)8 << capacity_log2;
}

int pk_attach_stamps(pk_ctx *ctx, uint64_t *stamps_dev, size_t stamps_bytes, pk_stream stream) {
    if (!ctx) return PK_ERR_ARG;
    if (!stamps_dev) {
        ctx->stamps = nullptr;
        return PK_OK;
    }
    if (!aligned16(stamps_dev) || stamps_bytes < pk_stamps_bytes(ctx->capacity_log2)) return PK_ERR_ARG;
    if (cudaMemsetAsync(stamps_dev, 0, pk_stamps_bytes(ctx->capacity_log2), reinterpret_cast<cudaStream_t>(stream)) !=
        cudaSuccess)
        return PK_ERR_CUDA;
    ctx->stamps = reinterpret_cast<unsigned long long *>(stamps_dev);
    return PK_OK;
}

size_t pk_evict_scratch_bytes(uint32_t capacity_log2) {
    if (capacity_log2 < 1 || capacity_log2 > 31) return 0;
    return (size_t)pk_evict_scratch_bytes_impl(1ull << capacity_log2);
}

int pk_evict(pk_ctx *ctx, uint64_t budget, uint64_t keep, void *scratch_dev, size_t scratch_bytes,
             uint32_t *evicted_slots_dev, uint64_t evicted_cap, uint64_t *n_evicted_dev, int32_t *status_dev,
             pk_stream stream) {
    if (!ctx || !ctx->stamps || keep > budget || !scratch_dev || !aligned16(scratch_dev)) return PK_ERR_ARG;
    if (scratch_bytes < pk_evict_scratch_bytes_impl(ctx->capacity)) return PK_ERR_ARG;
    if (!aligned(evicted_slots_dev, 4) || !aligned(n_evicted_dev, 8) || !aligned(status_dev, 4)) return PK_ERR_ARG;
    return cuda_rc(pk_launch_evict(ctx, budget, keep, scratch_dev, evicted_slots_dev,
                                   evicted_slots_dev ? evicted_cap : 0,
                                   reinterpret_cast<unsigned long long *>(n_evicted_dev), status_dev,
                                   reinterpret_cast<cudaStream_t>(stream)));
}

int pk_evict_barrier_timeout_test(pk_ctx *ctx, uint64_t budget, void *scratch_dev, size_t scratch_bytes,
                                  uint32_t spin_limit, int32_t *status_dev, pk_stream stream) {
    if (!ctx || !ctx->stamps || !scratch_dev || !aligned16(scratch_dev) || !status_dev || spin_limit == 0)
        return PK_ERR_ARG;
    if (scratch_bytes < pk_evict_scratch_bytes_impl(ctx->capacity) || !aligned(status_dev, 4)) return PK_ERR_ARG;
    return cuda_rc(pk_launch_evict(ctx, budget, budget, scratch_dev, nullptr, 0, nullptr, status_dev,
                                   reinterpret_cast<cudaStream_t>(stream), spin_limit, true));
}

int pk_key_string(const uint8_t key16[16], char out[22]) {
    if (!key16 || !out) return PK_ERR_ARG;
    base64_16(key16, out);
    return PK_OK;
}

int pk_model_tag(const pk_descriptor *desc, char out[22]) {
    if (!out) return PK_ERR_ARG;
    uint8_t dw[32];
    const int rc = pk_worker_digest(desc, dw);
    if (rc != PK_OK) return rc;
    base64_16(dw, out);
    return PK_OK;
}

int pk_key_strings(const uint8_t *keys_dev, uint64_t n, const char *prefix, uint32_t prefix_len, uint32_t width,
                   char *out_dev, pk_stream stream) {
    if (width > PK_KEY_STRING_MAX_WIDTH || prefix_len + PK_KEY_STRING_CHARS > width) return PK_ERR_ARG;
    if (prefix_len && !prefix) return PK_ERR_ARG;
    if (n == 0) return PK_OK;
    if (!keys_dev || !out_dev || !aligned16(keys_dev) || !aligned16(out_dev)) return PK_ERR_ARG;
    return cuda_rc(pk_launch_key_strings(keys_dev, n, reinterpret_cast<const uint8_t *>(prefix), prefix_len, width,
                                         reinterpret_cast<uint8_t *>(out_dev), reinterpret_cast<cudaStream_t>(stream)));
}

int pk_derive_lookup_store(pk_ctx *ctx, const int32_t *tokens_dev, uint64_t n_tokens, const int64_t *tok_off_dev,
                           uint32_t R, const uint32_t *desc_idx_dev, const uint8_t *enc_dev, uint64_t enc_bytes,
                           const int64_t *enc_off_dev, uint32_t D, uint8_t *digests_dev, int64_t *key_off_dev,
                           uint8_t *keys_dev, uint64_t key_capacity, const uint32_t *slots_new_dev,
                           int32_t *hit_chunks_dev, uint32_t *slots_dev, int32_t *result_dev, uint32_t *slot_out_dev,
                           int32_t *status_dev, pk_stream stream) {
    // the checks of pk_derive_keys_enc ...
    if (!ctx || !tok_off_dev || !key_off_dev) return PK_ERR_ARG;
    if (n_tokens && !tokens_dev) return PK_ERR_ARG;
    if (R && (!desc_idx_dev || D == 0 || !hit_chunks_dev)) return PK_ERR_ARG;
    if (D && (!enc_off_dev || !digests_dev || !aligned16(digests_dev) || !aligned(enc_off_dev, 8))) return PK_ERR_ARG;
    if (enc_bytes && !enc_dev) return PK_ERR_ARG;
    if (key_capacity < n_tokens / ctx->chunk_tokens) return PK_ERR_ARG;
    if (key_capacity && (!keys_dev || !aligned16(keys_dev))) return PK_ERR_ARG;
    if (!aligned(tokens_dev, 4) || !aligned(tok_off_dev, 8) || !aligned(desc_idx_dev, 4) || !aligned(key_off_dev, 8))
        return PK_ERR_ARG;
    // ... and of pk_lookup_store
    if (key_capacity && (!slots_new_dev || !slots_dev || !result_dev || !slot_out_dev)) return PK_ERR_ARG;
    if (key_capacity > (uint64_t)0x7fffffff * 64 || key_capacity >= 0xffffffffull) return PK_ERR_ARG;
    if (!aligned(hit_chunks_dev, 4) || !aligned(slots_new_dev, 4) || !aligned(slots_dev, 4) || !aligned(result_dev, 4) ||
        !aligned(slot_out_dev, 4))
        return PK_ERR_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = pk_launch_derive_enc(ctx, tokens_dev, n_tokens, tok_off_dev, R, desc_idx_dev, enc_dev, enc_bytes,
                                         D ? enc_off_dev : nullptr, D, digests_dev, key_off_dev, keys_dev, key_capacity,
                                         status_dev, s);
    if (e != cudaSuccess) return PK_ERR_CUDA;
    const unsigned long long epoch = ++ctx->epoch;
    return cuda_rc(pk_launch_lookup_store(ctx, epoch, keys_dev, slots_new_dev, key_off_dev, R, key_capacity,
                                          hit_chunks_dev, slots_dev, result_dev, slot_out_dev, status_dev, s));
}

int pk_compare_pages(const uint32_t *slots_dev, const uint8_t *pages_dev, const uint8_t *ref_pages_dev, uint64_t n,
                     uint64_t n_ref, uint64_t page_bytes, int32_t *verdict_dev, uint64_t *counts_dev,
                     int32_t *status_dev, pk_stream stream) {
    if (n == 0) return PK_OK;
    if (!slots_dev || !pages_dev || !verdict_dev || !counts_dev || (n_ref && !ref_pages_dev)) return PK_ERR_ARG;
    if (page_bytes == 0 || page_bytes % 16 || !aligned16(pages_dev) || !aligned16(ref_pages_dev) ||
        !aligned(slots_dev, 4) || !aligned(verdict_dev, 4) || !aligned(counts_dev, 8))
        return PK_ERR_ARG;
    return cuda_rc(pk_launch_compare_pages(slots_dev, pages_dev, ref_pages_dev, n, n_ref, page_bytes, verdict_dev,
                                           reinterpret_cast<unsigned long long *>(counts_dev), status_dev,
                                           reinterpret_cast<cudaStream_t>(stream)));
}

size_t pk_content_scratch_bytes(uint64_t n_bytes) { return (size_t)pk_content_scratch_bytes_impl(n_bytes); }

int pk_content_digest(const uint8_t *bytes_dev, uint64_t n_bytes, uint8_t *scratch_dev, size_t scratch_bytes,
                      uint8_t *top_dev, pk_stream stream) {
    if ((n_bytes && !bytes_dev) || !scratch_dev || !top_dev) return PK_ERR_ARG;
    if (!aligned16(bytes_dev) || !aligned16(scratch_dev) || !aligned16(top_dev)) return PK_ERR_ARG;
    if (scratch_bytes < pk_content_scratch_bytes_impl(n_bytes)) return PK_ERR_ARG;
    return cuda_rc(pk_launch_content_digest(bytes_dev, n_bytes, scratch_dev, top_dev,
                                            reinterpret_cast<cudaStream_t>(stream)));
}

size_t pk_content_scratch_bytes_batch(const uint64_t *n_bytes, uint32_t n) {
    if (n && !n_bytes) return 0;
    uint64_t total = 0;
    for (uint32_t j = 0; j < n; ++j) total += (pk_content_scratch_bytes_impl(n_bytes[j]) + 15) & ~15ull;
    return (size_t)total;
}

int pk_content_digests(const uint8_t *const *bytes_dev, const uint64_t *n_bytes, uint32_t n, uint8_t *scratch_dev,
                       size_t scratch_bytes, uint8_t *tops_dev, pk_stream stream) {
    if (n == 0) return PK_OK;
    if (!bytes_dev || !n_bytes || !scratch_dev || !tops_dev || !aligned16(scratch_dev) || !aligned16(tops_dev))
        return PK_ERR_ARG;
    std::vector<uint64_t> off(n);
    uint64_t total = 0;
    for (uint32_t j = 0; j < n; ++j) {
        if ((n_bytes[j] && !bytes_dev[j]) || !aligned16(bytes_dev[j])) return PK_ERR_ARG;
        off[j] = total;
        total += (pk_content_scratch_bytes_impl(n_bytes[j]) + 15) & ~15ull;
    }
    if (scratch_bytes < total) return PK_ERR_ARG;
    return cuda_rc(pk_launch_content_digests(bytes_dev, n_bytes, n, scratch_dev, off.data(), tops_dev,
                                             reinterpret_cast<cudaStream_t>(stream)));
}

int pk_tensor_identity(const pk_bytes *name, const pk_bytes *dtype, const int64_t *shape, uint32_t ndim,
                       uint64_t n_bytes, const uint8_t top[32], uint8_t out[32]) {
    if (!name || !dtype || (ndim && !shape) || !top || !out) return PK_ERR_ARG;
    std::string f[2];
    int rc;
    if ((rc = opaque(*name, &f[0])) != PK_OK) return rc;
    if ((rc = opaque(*dtype, &f[1])) != PK_OK) return rc;
    std::string dims, len;
    for (uint32_t k = 0; k < ndim; ++k) {
        put_le32(&dims, (uint32_t)((uint64_t)shape[k] & 0xffffffffu));
        put_le32(&dims, (uint32_t)((uint64_t)shape[k] >> 32));
    }
    put_le32(&len, (uint32_t)(n_bytes & 0xffffffffu));
    put_le32(&len, (uint32_t)(n_bytes >> 32));
    std::string enc;
    put_le32(&enc, 5u);
    for (const std::string *x : {&f[0], &f[1], &dims, &len}) {
        put_le32(&enc, (uint32_t)x->size());
        enc.append(*x);
    }
    put_le32(&enc, 32u);
    enc.append(reinterpret_cast<const char *>(top), 32);
    pk::sha256_bytes(reinterpret_cast<const uint8_t *>(enc.data()), enc.size(), out);
    return PK_OK;
}

int pk_adapter_identity(const uint8_t *tensor_ids, uint32_t n_tensors, const pk_bytes *config, uint32_t n_config,
                        uint8_t out[32]) {
    if ((n_tensors && !tensor_ids) || (n_config && !config) || !out) return PK_ERR_ARG;
    std::string cfg;
    put_le32(&cfg, n_config);
    for (uint32_t k = 0; k < n_config; ++k) {
        std::string x;
        const int rc = opaque(config[k], &x);
        if (rc != PK_OK) return rc;
        put_le32(&cfg, (uint32_t)x.size());
        cfg.append(x);
    }
    std::string enc;
    put_le32(&enc, 1u + n_tensors);
    put_le32(&enc, (uint32_t)cfg.size());
    enc.append(cfg);
    for (uint32_t t = 0; t < n_tensors; ++t) {
        put_le32(&enc, 32u);
        enc.append(reinterpret_cast<const char *>(tensor_ids + 32ull * t), 32);
    }
    pk::sha256_bytes(reinterpret_cast<const uint8_t *>(enc.data()), enc.size(), out);
    return PK_OK;
}

int pk_table_save(pk_ctx *ctx, void *dst, size_t dst_bytes, pk_stream stream) {
    if (!ctx || !dst) return PK_ERR_ARG;
    const size_t tb = pk_table_bytes(ctx->capacity_log2);
    if (dst_bytes < tb + 64) return PK_ERR_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(dst, ctx->table, tb, cudaMemcpyDefault, s) != cudaSuccess ||
        cudaMemcpyAsync(static_cast<uint8_t *>(dst) + tb, ctx->counter_dev, sizeof(unsigned long long),
                        cudaMemcpyDefault, s) != cudaSuccess)
        return PK_ERR_CUDA;
    return PK_OK;
}

int pk_table_load(pk_ctx *ctx, const void *src, size_t src_bytes, pk_stream stream) {
    if (!ctx || !src) return PK_ERR_ARG;
    const size_t tb = pk_table_bytes(ctx->capacity_log2);
    if (src_bytes < tb + 64) return PK_ERR_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (ctx->epoch < 1) ctx->epoch = 1;
    if (ctx->stamps && cudaMemsetAsync(ctx->stamps, 0, 8ull * ctx->capacity, s) != cudaSuccess) return PK_ERR_CUDA;
    cudaPointerAttributes attr;
    const bool on_device = cudaPointerGetAttributes(&attr, src) == cudaSuccess &&
                           (attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged) &&
                           aligned16(src);
    if (!on_device) cudaGetLastError();  // (a host pointer may leave an error from the query)
    if (on_device) return cuda_rc(pk_launch_load_table(ctx, src, s));  // one pass, copy and mark
    if (cudaMemcpyAsync(ctx->table, src, tb, cudaMemcpyDefault, s) != cudaSuccess ||
        cudaMemcpyAsync(ctx->counter_dev, static_cast<const uint8_t *>(src) + tb, sizeof(unsigned long long),
                        cudaMemcpyDefault, s) != cudaSuccess)
        return PK_ERR_CUDA;
    return cuda_rc(pk_launch_mark_loaded(ctx, s));
}

int pk_store_noalloc(const pk_config *cfg, const uint8_t *keys_dev, const uint32_t *slots_dev, uint64_t n,
                     const int64_t *key_off_dev, const int32_t *hit_chunks_dev, uint32_t R, int32_t *result_dev,
                     uint32_t *slot_out_dev, int32_t *status_dev, pk_stream stream) {
    if (!cfg || !cfg->table_dev || !aligned16(cfg->table_dev)) return PK_ERR_ARG;
    const size_t need = pk_table_bytes(cfg->capacity_log2);
    if (need == 0 || cfg->table_bytes < need) return PK_ERR_CAPACITY;
    if ((key_off_dev == nullptr) != (hit_chunks_dev == nullptr)) return PK_ERR_ARG;
    if (n > PK_NOALLOC_MAX_ENTRIES) return PK_ERR_TOO_LARGE;
    if (n == 0) return PK_OK;
    if (!keys_dev || !aligned16(keys_dev) || !slots_dev || !result_dev || !slot_out_dev) return PK_ERR_ARG;
    if (!aligned(slots_dev, 4) || !aligned(result_dev, 4) || !aligned(slot_out_dev, 4) || !aligned(key_off_dev, 8) ||
        !aligned(hit_chunks_dev, 4))
        return PK_ERR_ARG;
    const uint64_t capacity = 1ull << cfg->capacity_log2;
    const uint32_t max_probe =
        (cfg->max_probe == 0 || cfg->max_probe > capacity) ? (uint32_t)capacity : cfg->max_probe;
    return cuda_rc(pk_launch_store_noalloc(static_cast<pk_entry *>(cfg->table_dev), cfg->capacity_log2, max_probe,
                                           keys_dev, slots_dev, n, key_off_dev, hit_chunks_dev, R, result_dev,
                                           slot_out_dev, status_dev, reinterpret_cast<cudaStream_t>(stream)));
}

int pk_entries(pk_ctx *ctx, uint64_t *count, pk_stream stream) {
    if (!ctx || !count) return PK_ERR_ARG;
    unsigned long long v = 0;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(&v, ctx->counter_dev, sizeof v, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return PK_ERR_CUDA;
    *count = v;
    return PK_OK;
}

const char *pk_strerror(int code) {
    switch (code) {
        case PK_OK: return "ok";
        case PK_ERR_ARG: return "invalid argument";
        case PK_ERR_CAPACITY: return "capacity not a power of two in [2, 2^31] or table buffer too small";
        case PK_ERR_UNRESOLVED: return "weight precision or KV format is empty or unresolved (auto)";
        case PK_ERR_FIELD_TOO_LONG: return "descriptor field longer than PK_MAX_FIELD_BYTES";
        case PK_ERR_TABLE_FULL: return "table full";
        case PK_ERR_PROBE_LIMIT: return "probe limit reached";
        case PK_ERR_RESERVED_KEY: return "key prefix is the reserved all-zero value";
        case PK_ERR_CUDA: return "CUDA runtime error";
        case PK_ERR_TIMEOUT: return "a bounded device-wide wait gave up (the table is unspecified)";
        case PK_ERR_TOO_LARGE: return "more entries than the allocation-free store's scratch holds (PK_NOALLOC_MAX_ENTRIES)";
        default: return "unknown status";
    }
}

}  // extern "C"
