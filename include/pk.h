/*
 * pk.h -- C ABI of libpk: provenance-bound KV-cache keys on one GPU.
 *
 * The paper ("Preserving Provenance in Shared KV Caches for LLM Serving")
 * requires a shared KV tier's key to be injective over every declared
 * provenance dimension (Def. 2, Eqs. 1 and 2) and realises it as
 *     Key(x, c) = f(x, H(enc(id_1(c(d_1)), ..., id_n(c(d_n)))))      (Eq. 3)
 * This library computes that key for a batch of requests and keeps a
 * GPU-resident table of key prefixes, with
 *     H   = SHA-256,  d = H(enc(canonical descriptor))
 *     f   = chained per-chunk digest:
 *           c_i = SHA-256(int32 little-endian bytes of tokens[iC, (i+1)C))
 *           k_i = SHA-256(k_{i-1} || d || c_i),   k_{-1} = 32 zero bytes
 * over the floor(T/C) full chunks of each request (a partial trailing chunk
 * gets no key; Sec. 4.4).  The table maps the first 16 bytes of k_i (the
 * 128-bit digest width of Sec. 5.3) to a uint32 chunk slot.  Lookup returns
 * each request's longest all-hit prefix; store inserts the misses (Sec. 2.1:
 * on a local miss the connector queries the store; a hit skips that prefill,
 * a miss computes and writes new state).  Lookup and store consume keys from
 * one pk_derive_keys call, so both sites derive keys from the same
 * descriptor value (Sec. 5.3, "Cross-site consistency").
 *
 * Conventions for every call
 *   - Returns PK_OK (0) or a negative PK_ERR_* code.  A host-detected error
 *     returns before anything is enqueued and leaves the table unchanged.
 *   - "_dev" pointers are device memory owned by the caller; the library
 *     allocates no device memory except a small fixed block in pk_init.
 *   - All device work is enqueued asynchronously on the given stream
 *     (NULL = legacy default stream).  Errors found on the device are written
 *     to the caller's int32 status word *status_dev (first error wins; the
 *     caller zeroes it and reads it after synchronising).  After a device
 *     error the call's outputs are unspecified, but no access leaves the
 *     caller's buffers and no wait is unbounded.
 *   - A context is not thread-safe; calls on one context must be ordered.
 */
#ifndef PK_H_
#define PK_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
#define PK_OK 0
#define PK_ERR_ARG (-1)            /* null / misaligned pointer, bad size, bad offsets or index */
#define PK_ERR_CAPACITY (-2)       /* capacity not a power of two in [2, 2^31], or table too small */
#define PK_ERR_UNRESOLVED (-3)     /* precision or KV format empty or "auto" (Sec. 5.3) */
#define PK_ERR_FIELD_TOO_LONG (-4) /* a descriptor field over PK_MAX_FIELD_BYTES */
#define PK_ERR_TABLE_FULL (-5)     /* insertion would leave no empty slot */
#define PK_ERR_PROBE_LIMIT (-6)    /* probe sequence longer than max_probe */
#define PK_ERR_RESERVED_KEY (-7)   /* key prefix is all zero (the empty marker), p = 2^-128 */
#define PK_ERR_CUDA (-8)           /* a CUDA runtime call or launch failed */
#define PK_ERR_TOO_LARGE (-9)      /* n above PK_NOALLOC_MAX_ENTRIES (pk_store_noalloc only) */
#define PK_ERR_TIMEOUT (-10)       /* a bounded device-wide wait gave up (pk_evict); table unspecified */

/* Per-entry store results (int32). Negative values are the error codes above. */
#define PK_STORE_SKIPPED 0         /* not in a miss range (range mode) */
#define PK_STORE_INSERTED 1        /* new key; the entry's own slot was stored */
#define PK_STORE_PRESENT 2         /* key already present (or an earlier duplicate in the batch won) */

#define PK_PAGE_ABSENT 0           /* pk_compare_pages: the key has no reference page */
#define PK_PAGE_EQUAL 1            /* equal key, equal page bytes */
#define PK_PAGE_DIFFERS 2          /* equal key, differing page bytes: an omitted binding */

#define PK_NO_SLOT 0xFFFFFFFFu     /* lookup miss; not a storable slot value */
#define PK_MAX_FIELD_BYTES 4096u
#define PK_KEY_BYTES 32u           /* one full key k_i */
#define PK_PREFIX_BYTES 16u        /* table key = first 16 bytes of k_i */
#define PK_ENTRY_BYTES 32u         /* one table entry in device memory */

typedef struct pk_ctx pk_ctx;
/* Same type as cudaStream_t. */
typedef struct CUstream_st *pk_stream;

/* A byte string; p may be NULL when len == 0. */
typedef struct {
    const uint8_t *p;
    uint32_t len;
} pk_bytes;

/* One provenance descriptor: registry v1 in encoding order (Sec. 5.1 dimensions
 * plus the model identity, Sec. 5.3), then optional appended dimensions
 * (Prop. 1: appending a well-formed dimension preserves the contract).
 * Empty adapter_id / salt mean "none".  weight_precision and kv_format must be
 * resolved values (ASCII case-insensitive; bfloat16->bf16, float16|half->fp16,
 * float32|float->fp32, float8_e4m3fn->fp8_e4m3, float8_e5m2->fp8_e5m2; any
 * other spelling is kept as written).  Other fields are opaque bytes. */
typedef struct {
    pk_bytes model_id;
    pk_bytes weight_precision;
    pk_bytes weight_version;
    pk_bytes adapter_id;
    pk_bytes kv_format;
    pk_bytes salt;
    const pk_bytes *extra; /* n_extra appended dimension identities, or NULL */
    uint32_t n_extra;
} pk_descriptor;

typedef struct {
    uint32_t chunk_tokens;  /* C >= 1 */
    uint32_t capacity_log2; /* table capacity = 2^capacity_log2, 1..31 */
    uint32_t max_probe;     /* probe sequence bound per key; 0 = capacity */
    void *table_dev;        /* caller-owned, 16-byte aligned */
    size_t table_bytes;     /* >= pk_table_bytes(capacity_log2) */
} pk_config;

/* Bytes of device memory a table of 2^capacity_log2 entries needs (0 if out of range). */
size_t pk_table_bytes(uint32_t capacity_log2);

/* Create a context bound to the caller's table and clear the table (all
 * entries empty) on `stream`.  Allocates one small device block (entry
 * counter).  *out is NULL on error.  Errors: PK_ERR_ARG, PK_ERR_CAPACITY,
 * PK_ERR_CUDA. */
int pk_init(pk_ctx **out, const pk_config *cfg, pk_stream stream);

/* Release the context (not the caller's table).  Synchronises nothing;
 * the caller must not destroy a context with work still in flight. */
int pk_destroy(pk_ctx *ctx);

/* Host.  Canonicalise one descriptor and write enc = LE32(field count) ||
 * (LE32(len) || bytes) per field (Sec. 5.2: injective, length-prefixed) into
 * out[0, cap).  *len receives the encoded size (also when cap is too small,
 * in which case PK_ERR_ARG is returned).  Errors: PK_ERR_ARG,
 * PK_ERR_UNRESOLVED, PK_ERR_FIELD_TOO_LONG. */
int pk_descriptor_encode(const pk_descriptor *desc, uint8_t *out, size_t cap, size_t *len);

/* Host.  Encode D descriptors back to back; enc_off (D+1 entries) receives the
 * byte offsets.  Same errors as pk_descriptor_encode (first failing one). */
int pk_descriptors_encode(const pk_descriptor *descs, uint32_t D, uint8_t *out, size_t cap,
                          int64_t *enc_off);

/* Host.  d = SHA-256(enc(canonical descriptor)) (Eq. 3, H over enc). */
int pk_descriptor_digest(const pk_descriptor *desc, uint8_t out[32]);

/* Host.  Two-level variant: the worker-level and request-level halves of the
 * descriptor bound through separate digests (Sec. 2.2), the worker half
 * digested once over resolved values (Sec. 5.3, worker-level digest), the
 * request half inert when it is empty (Sec. 5.3, request-level tags):
 *   pk_worker_digest:  d_w = SHA-256(enc_w), enc_w = LE32(4) || (LE32(len) ||
 *                      bytes) for model id, weight precision, weight version,
 *                      KV format (canonicalised as above); the descriptor's
 *                      adapter, salt and appended dimensions are ignored.
 *   pk_request_digest: d = d_w (worker, 32 bytes) when the descriptor has no
 *                      adapter, no salt and no appended dimension (such a
 *                      request keys exactly as the worker-only chain), else
 *                      d = SHA-256(d_w || SHA-256(enc_q)), enc_q = LE32(2 +
 *                      n_extra) || (LE32(len) || bytes) for adapter id, salt,
 *                      appended dimensions; the worker fields are ignored.
 * d replaces the single-digest d of pk_descriptor_digest as the digest of
 * pk_derive_keys.  Errors: PK_ERR_ARG, PK_ERR_UNRESOLVED (worker),
 * PK_ERR_FIELD_TOO_LONG. */
int pk_worker_digest(const pk_descriptor *desc, uint8_t out[32]);
int pk_request_digest(const uint8_t worker[32], const pk_descriptor *desc, uint8_t out[32]);
/* Host.  pk_request_digest for n descriptors of one worker: out[j*32, j*32+32)
 * for descs[j]; stops at the first error (its code is returned). */
int pk_request_digests(const uint8_t worker[32], const pk_descriptor *descs, uint32_t n, uint8_t *out);

/* Device.  digests_dev[j] = SHA-256(enc_dev[enc_off_dev[j], enc_off_dev[j+1]))
 * for j < D: the descriptor digests d of a batch (Eq. 3, H over enc), from
 * encodings produced by pk_descriptors_encode and copied to the device.
 * enc_dev holds enc_bytes bytes; enc_off_dev holds D+1 offsets; digests_dev:
 * D*32 bytes.  Device errors (offsets decreasing or beyond enc_bytes):
 * PK_ERR_ARG in *status_dev, that digest left unwritten. */
int pk_digest_descriptors(pk_ctx *ctx, const uint8_t *enc_dev, uint64_t enc_bytes,
                          const int64_t *enc_off_dev, uint32_t D, uint8_t *digests_dev,
                          int32_t *status_dev, pk_stream stream);

/* Device.  Key derivation for R requests: Key(x, c) = f(x, d) of Eq. 3
 * (Sec. 5.2), f being the chained per-chunk digest of the header (steps c_i
 * and k_i above), with keys only for full chunks (Sec. 4.4).
 *   tokens_dev   int32[n_tokens]
 *   tok_off_dev  int64[R+1], non-decreasing, tok_off[R] <= n_tokens;
 *                request r = tokens[tok_off[r], tok_off[r+1])
 *   desc_idx_dev uint32[R] < D;  digests_dev uint8[D*32] (16-byte aligned)
 *   key_off_dev  OUT int64[R+1]: key_off[0] = 0,
 *                key_off[r+1] = key_off[r] + floor((tok_off[r+1]-tok_off[r]) / C)
 *   keys_dev     OUT uint8[key_capacity*32] (16-byte aligned): key j of
 *                request r at index key_off[r] + j.  key_capacity must be at
 *                least floor(n_tokens / C), which always suffices.
 * Any request layout is accepted (starts need not be aligned).  Device errors
 * (offsets not monotone or out of range, desc_idx >= D): PK_ERR_ARG in
 * *status_dev and key_off all zero. */
int pk_derive_keys(pk_ctx *ctx, const int32_t *tokens_dev, uint64_t n_tokens,
                   const int64_t *tok_off_dev, uint32_t R, const uint32_t *desc_idx_dev,
                   const uint8_t *digests_dev, uint32_t D, int64_t *key_off_dev,
                   uint8_t *keys_dev, uint64_t key_capacity, int32_t *status_dev,
                   pk_stream stream);

/* Device.  pk_digest_descriptors and pk_derive_keys in one call: the
 * descriptor encodings (as for pk_digest_descriptors) are hashed inside the
 * key-derivation launch, alongside the chunk digests that do not depend on
 * them, and the digests d are also written to digests_dev (D*32 bytes,
 * 16-byte aligned).  Other arguments, outputs and errors as pk_derive_keys;
 * D may be 0 only when R is 0. */
int pk_derive_keys_enc(pk_ctx *ctx, const int32_t *tokens_dev, uint64_t n_tokens,
                       const int64_t *tok_off_dev, uint32_t R, const uint32_t *desc_idx_dev,
                       const uint8_t *enc_dev, uint64_t enc_bytes, const int64_t *enc_off_dev,
                       uint32_t D, uint8_t *digests_dev, int64_t *key_off_dev, uint8_t *keys_dev,
                       uint64_t key_capacity, int32_t *status_dev, pk_stream stream);

/* Device.  The lookup of Sec. 2.1 (on a local miss the connector queries
 * the shared store, and a hit skips that prefill), keyed by the 128-bit
 * prefix of each k_i (Sec. 5.3: the digest is kept at 128 bits).  Probe the
 * table for every key of a pk_derive_keys result.
 *   slots_dev       OUT uint32[key_capacity]: slot of key i, or PK_NO_SLOT
 *   hit_chunks_dev  OUT int32[R]: h_r = the largest j such that keys 0..j-1 of
 *                   request r are all present (the first miss ends the prefix);
 *                   the keys to store are those of [h_r, n_r)
 * The table is read as of the start of the call.  Device errors:
 * PK_ERR_PROBE_LIMIT (that key reads as a miss). */
int pk_lookup(pk_ctx *ctx, const uint8_t *keys_dev, const int64_t *key_off_dev, uint32_t R,
              uint64_t key_capacity, int32_t *hit_chunks_dev, uint32_t *slots_dev,
              int32_t *status_dev, pk_stream stream);

/* Device.  The store of Sec. 2.1 (on a miss the connector computes the
 * chunk's state and writes it to the shared store under the same key), over
 * 128-bit key prefixes (Sec. 5.3).  Insert-if-absent of (prefix of keys_dev[e], slots_dev[e]), with
 * the outcome of processing the entries one by one in index order: an absent
 * key is inserted with its own slot (PK_STORE_INSERTED); a key already in the
 * table, or inserted by a lower index of the same call, keeps the existing
 * slot (PK_STORE_PRESENT).  slot_out_dev[e] receives the slot now bound to the
 * key (PK_NO_SLOT for skipped or failed entries).
 *   list mode  (key_off_dev == NULL, hit_chunks_dev == NULL): entries 0..n-1
 *   range mode (both given, R requests): only the miss ranges
 *              [key_off[r] + hit_chunks[r], key_off[r+1]) of a pk_lookup
 *              result; n = key_capacity; other entries get PK_STORE_SKIPPED.
 * keys_dev: n*32 bytes (only the first 16 of each used), 16-byte aligned;
 * slots_dev: uint32[n], values != PK_NO_SLOT; result_dev: int32[n];
 * slot_out_dev: uint32[n] (required: also holds intermediate positions).
 * Per-entry errors: PK_ERR_RESERVED_KEY, PK_ERR_ARG (slot == PK_NO_SLOT),
 * PK_ERR_TABLE_FULL, PK_ERR_PROBE_LIMIT; the first one also goes to
 * *status_dev.  Capacity: the table never holds more than capacity - 1
 * entries (one always stays empty, so every probe ends), and refusals follow
 * the index order too: with `room` = capacity - 1 - entries at the start of
 * the call, the first `room` distinct new keys (ranked by their lowest
 * index) are inserted and every entry of a later new key gets
 * PK_ERR_TABLE_FULL.  A call that may not fit (entries + n >= capacity) adds
 * a pass over its new keys, in index order when they do not all fit. */
int pk_store(pk_ctx *ctx, const uint8_t *keys_dev, const uint32_t *slots_dev, uint64_t n,
             const int64_t *key_off_dev, const int32_t *hit_chunks_dev, uint32_t R,
             int32_t *result_dev, uint32_t *slot_out_dev, int32_t *status_dev, pk_stream stream);

/* Device.  pk_lookup followed by pk_store in range mode, in one pass over
 * the keys (Sec. 2.1: the connector looks the chunks up, and a miss computes
 * and writes new state).  Every key of the batch is inserted if absent, keys
 * inserted earlier in the same call counting as absent, so each key's probe
 * sequence is walked once:
 *   slots_dev, hit_chunks_dev  OUT as pk_lookup (the table as of the start
 *                              of the call)
 *   result_dev, slot_out_dev   OUT as pk_store in range mode over the miss
 *                              ranges [key_off[r] + h_r, key_off[r+1]) with
 *                              slots slots_new_dev; other entries
 *                              PK_STORE_SKIPPED
 * keys_dev as pk_lookup (16-byte aligned); slots_new_dev, slots_dev,
 * result_dev, slot_out_dev: key_capacity entries of 4 bytes.  A key whose new
 * slot is PK_NO_SLOT is only looked up (PK_ERR_ARG if it lies in its miss
 * range).  Results equal those of the two calls; device errors as the two
 * calls, the first one observed going to *status_dev. */
int pk_lookup_store(pk_ctx *ctx, const uint8_t *keys_dev, const uint32_t *slots_new_dev, const int64_t *key_off_dev,
                    uint32_t R, uint64_t key_capacity, int32_t *hit_chunks_dev, uint32_t *slots_dev,
                    int32_t *result_dev, uint32_t *slot_out_dev, int32_t *status_dev, pk_stream stream);

/* Device.  The whole hot path in one call (a0-a4): pk_derive_keys_enc
 * followed by pk_lookup_store on its keys, enqueued together.  Arguments as
 * the two calls (tokens ... key_capacity as pk_derive_keys_enc; slots_new_dev,
 * hit_chunks_dev, slots_dev, result_dev, slot_out_dev as pk_lookup_store);
 * outputs, results and device errors equal those of the two calls (one store
 * call number); all host checks run before anything is enqueued. */
int pk_derive_lookup_store(pk_ctx *ctx, const int32_t *tokens_dev, uint64_t n_tokens, const int64_t *tok_off_dev,
                           uint32_t R, const uint32_t *desc_idx_dev, const uint8_t *enc_dev, uint64_t enc_bytes,
                           const int64_t *enc_off_dev, uint32_t D, uint8_t *digests_dev, int64_t *key_off_dev,
                           uint8_t *keys_dev, uint64_t key_capacity, const uint32_t *slots_new_dev,
                           int32_t *hit_chunks_dev, uint32_t *slots_dev, int32_t *result_dev, uint32_t *slot_out_dev,
                           int32_t *status_dev, pk_stream stream);

/* Device.  The comparison step of the store-side differential omission test
 * (Sec. 6.3, omission detection; Eq. 4): a worker's keys joined to a
 * reference worker's by pk_lookup on a table holding the reference keys
 * (slot = index of the reference page), then each joined page compared byte
 * for byte.
 *   slots_dev      uint32[n]: the reference page of key j, or PK_NO_SLOT
 *   pages_dev      n pages of page_bytes (the worker's page of key j)
 *   ref_pages_dev  n_ref pages of page_bytes
 *   verdict_dev    OUT int32[n]: PK_PAGE_ABSENT, PK_PAGE_EQUAL or PK_PAGE_DIFFERS
 *   counts_dev     IN/OUT uint64[3]: counts_dev[v] += keys with verdict v
 *                  (zero it first for this call's counts)
 * page_bytes: a positive multiple of 16; page buffers 16-byte aligned.  Every
 * joined pair is read in full.  Device errors: a slot >= n_ref (PK_ERR_ARG in
 * *status_dev; that key reads as PK_PAGE_ABSENT). */
int pk_compare_pages(const uint32_t *slots_dev, const uint8_t *pages_dev, const uint8_t *ref_pages_dev, uint64_t n,
                     uint64_t n_ref, uint64_t page_bytes, int32_t *verdict_dev, uint64_t *counts_dev,
                     int32_t *status_dev, pk_stream stream);

/* Content identity of large byte buffers (Sec. 5.3: an adapter is bound by an
 * identity of its contents, every tensor's name, dtype, shape and bytes with
 * the meaningful configuration fields; Sec. 5.1 leaves the identity function
 * open as long as it is injective and stable).  One SHA-256 stream over a
 * tensor is serial, so the bytes are reduced by a fixed-shape tree instead:
 * every level hashes each 1 KiB block of the level below (the last block
 * zero-padded; an empty buffer is one zero block), down to one digest, the
 * "top".  The shape depends only on the byte length, which the tensor
 * identity binds.
 *   pk_content_scratch_bytes: device scratch pk_content_digest needs for n_bytes.
 *   pk_content_digest (device): top_dev (32 bytes) = the tree top of
 *                     bytes_dev[0, n_bytes); bytes_dev, scratch_dev, top_dev
 *                     16-byte aligned.  Errors: PK_ERR_ARG (host), PK_ERR_CUDA.
 *   pk_tensor_identity (host): SHA-256(enc(name, dtype, shape as LE64 each,
 *                     LE64(n_bytes), top)).
 *   pk_adapter_identity (host): SHA-256(enc(enc(config fields), tensor
 *                     identity_0, ..., identity_{n-1})), the tensors in the
 *                     order given (sort them by name for a stable identity). */
size_t pk_content_scratch_bytes(uint64_t n_bytes);
int pk_content_digest(const uint8_t *bytes_dev, uint64_t n_bytes, uint8_t *scratch_dev, size_t scratch_bytes,
                      uint8_t *top_dev, pk_stream stream);
/* The same for n buffers at once (an adapter's tensors): tops_dev[32 j ..]
 * = the tree top of bytes_dev[j][0, n_bytes[j]).  bytes_dev and n_bytes are
 * host arrays of n entries (device pointers, 16-byte aligned); every tree
 * level of all the buffers (128 at a time) is one launch, so a call costs
 * about as many launches as its largest buffer has levels.  scratch_dev:
 * pk_content_scratch_bytes_batch(n_bytes, n) bytes, 16-byte aligned.
 * Errors: PK_ERR_ARG (host), PK_ERR_CUDA. */
size_t pk_content_scratch_bytes_batch(const uint64_t *n_bytes, uint32_t n);
int pk_content_digests(const uint8_t *const *bytes_dev, const uint64_t *n_bytes, uint32_t n, uint8_t *scratch_dev,
                       size_t scratch_bytes, uint8_t *tops_dev, pk_stream stream);
int pk_tensor_identity(const pk_bytes *name, const pk_bytes *dtype, const int64_t *shape, uint32_t ndim,
                       uint64_t n_bytes, const uint8_t top[32], uint8_t out[32]);
int pk_adapter_identity(const uint8_t *tensor_ids, uint32_t n_tensors, const pk_bytes *config, uint32_t n_config,
                        uint8_t out[32]);

/* Connector key strings (Sec. 5.3, connector integration).  A connector that
 * packs its key into a fixed-width text field carries the 128-bit digest as
 * PK_KEY_STRING_CHARS (22) base64 characters (RFC 4648, Sec. 4: alphabet
 * A-Z a-z 0-9 + /, big-endian 6-bit groups, the two "=" of padding dropped;
 * the last character encodes two bits followed by four zero bits) and the
 * model identity with the worker provenance as a fixed-length hash of the
 * same form, so the key's length does not depend on the model path.
 *   pk_key_string (host): out = base64 of key16[0, 16); no terminating NUL.
 *   pk_model_tag (host): out = pk_key_string of the first 16 bytes of the
 *                  worker digest d_w of pk_worker_digest (model id, weight
 *                  precision, weight version, KV format).  Errors as
 *                  pk_worker_digest.
 *   pk_key_strings (device): for i < n, row i of out_dev (bytes
 *                  [i*width, (i+1)*width)) = prefix[0, prefix_len) ||
 *                  base64 of keys_dev[i*32, i*32+16) || zero bytes up to the
 *                  row width.  keys_dev: n 32-byte keys of a pk_derive_keys
 *                  result (16-byte aligned); prefix: host bytes, the same for
 *                  every row (e.g. the connector's fixed fields and the model
 *                  tag), may be NULL when prefix_len == 0; out_dev: n*width
 *                  bytes, 16-byte aligned.  Requires prefix_len + 22 <= width
 *                  <= PK_KEY_STRING_MAX_WIDTH.  Errors (host, nothing
 *                  enqueued): PK_ERR_ARG; PK_ERR_CUDA. */
#define PK_KEY_STRING_CHARS 22u
#define PK_KEY_STRING_MAX_WIDTH 256u
int pk_key_string(const uint8_t key16[16], char out[22]);
int pk_model_tag(const pk_descriptor *desc, char out[22]);
int pk_key_strings(const uint8_t *keys_dev, uint64_t n, const char *prefix, uint32_t prefix_len, uint32_t width,
                   char *out_dev, pk_stream stream);

/* Eviction under a fixed budget (Sec. 6.5: provenance separation keeps one
 * copy per provenance, so a store of fixed size evicts more and thrashes once
 * the distinct working set exceeds it).  Budget mode keeps one last-use
 * stamp per table entry in a caller-owned array:
 *   stamp = (n << 32) | e, n the number of the store call on this context
 *           (pk_store and pk_lookup_store calls, counted from 1 after
 *           pk_init; after a pk_table_load the next call number is at least
 *           2), e the key's index in that call;
 * each pk_store and pk_lookup_store call raises it to its own for every key
 * of the call that was in the table at the start of the call, or is stored
 * by it with a valid slot (in pk_store, every entry with result
 * PK_STORE_INSERTED or PK_STORE_PRESENT).  pk_lookup reads only and stamps
 * nothing.  Entries stored before the stamps were attached (or before a
 * pk_table_load) have stamp 0.
 *   pk_stamps_bytes:  bytes of the stamp array (8 per entry; 0 if out of range).
 *   pk_attach_stamps: enable budget mode with stamps_dev (16-byte aligned,
 *                     >= pk_stamps_bytes) and zero it on `stream`; NULL
 *                     detaches.
 *   pk_evict_scratch_bytes: device scratch pk_evict needs (about 13.3
 *                     bytes per entry plus 8.5 KiB).
 *   pk_evict (device): when the table holds more than `budget` entries,
 *                     remove every entry whose stamp is at most v, the
 *                     (keep+1)-th largest stamp: the least recently used
 *                     entries down to `keep` (fewer remain only when stamps
 *                     tie at v, i.e. unstamped entries).  Otherwise nothing
 *                     changes.  The slots of the removed entries go to
 *                     evicted_slots_dev[0, *n_evicted_dev) in unspecified
 *                     order (evicted_slots_dev: uint32[evicted_cap] or NULL;
 *                     n_evicted_dev: uint64, 0 when nothing is removed, or
 *                     NULL); the entry count drops by their number.  Kept
 *                     entries keep their key, slot and stamp (their positions
 *                     may change).  Requires stamps attached, keep <= budget,
 *                     scratch_dev 16-byte aligned with scratch_bytes >=
 *                     pk_evict_scratch_bytes.  Device errors: more removals
 *                     than evicted_cap (PK_ERR_ARG; the extra slots are not
 *                     written); PK_ERR_TIMEOUT (table unspecified).  One
 *                     cooperative launch; within the budget it returns at
 *                     once. */
/* Test hook of pk_evict's bounded grid barriers (no paper counterpart): the
 * same launch as pk_evict(ctx, budget, budget, ...) with the barrier waits
 * bounded at spin_limit polls of about 100-200 ns (> 0; at most the default
 * of about a second) and CTA 0 withholding its arrival at the first barrier,
 * so that every other CTA's wait runs out.  Needs stamps attached and more
 * than `budget` entries in the table (else the kernel returns before the
 * barrier) and a table of at least 2^10 entries (two CTAs or more).  The
 * launch must end by itself with PK_ERR_TIMEOUT in *status_dev; the first
 * barrier precedes every write to the table and the stamps, so both are
 * unchanged, and the context stays usable.  Errors (host): PK_ERR_ARG,
 * PK_ERR_CUDA. */
int pk_evict_barrier_timeout_test(pk_ctx *ctx, uint64_t budget, void *scratch_dev, size_t scratch_bytes,
                                  uint32_t spin_limit, int32_t *status_dev, pk_stream stream);

size_t pk_stamps_bytes(uint32_t capacity_log2);
int pk_attach_stamps(pk_ctx *ctx, uint64_t *stamps_dev, size_t stamps_bytes, pk_stream stream);
size_t pk_evict_scratch_bytes(uint32_t capacity_log2);
int pk_evict(pk_ctx *ctx, uint64_t budget, uint64_t keep, void *scratch_dev, size_t scratch_bytes,
             uint32_t *evicted_slots_dev, uint64_t evicted_cap, uint64_t *n_evicted_dev, int32_t *status_dev,
             pk_stream stream);

/* Checkpoint (the shared store outlives workers, Sec. 2.1).  Asynchronous on
 * `stream`: copies the table and its entry count to dst (device or host
 * memory, dst_bytes >= pk_table_bytes(capacity_log2) + 64). */
int pk_table_save(pk_ctx *ctx, void *dst, size_t dst_bytes, pk_stream stream);

/* Resume: replace this context's table with one saved by pk_table_save from a
 * context of the same capacity (src: device or host memory, src_bytes >=
 * pk_table_bytes + 64).  Keys and slots are restored exactly; the entries
 * count as inserted before any later store call; attached stamps are
 * zeroed.  Asynchronous on `stream`. */
int pk_table_load(pk_ctx *ctx, const void *src, size_t src_bytes, pk_stream stream);

/* Device.  The insert-if-absent of pk_store for callers that cannot allocate
 * device memory and so cannot create a context (pk_init allocates the
 * context's entry counter): engines whose device memory is entirely owned by
 * their own pool with a fixed budget, and latency-critical paths that must
 * not enter the CUDA allocator (an allocation can synchronise the device).
 * The paper has no counterpart; this is an integration convenience.
 * The table is described by cfg (table_dev, table_bytes, capacity_log2,
 * max_probe; chunk_tokens is ignored) and must be all zero before its first
 * use (cudaMemset, or a table created by pk_init).  Arguments, results and
 * per-entry errors are those of pk_store, list or range mode.
 * No memory is allocated: the call's scratch (the table's entry count, the
 * latest call number in the table, the counts of the call's deferred and
 * claimed keys, and one 4-byte claim position per entry) is a fixed
 * file-scope device array of 40 + 4 * PK_NOALLOC_MAX_ENTRIES bytes
 * (about 1 MiB), held by every GPU that loads the library until the process
 * exits.  n > PK_NOALLOC_MAX_ENTRIES returns PK_ERR_TOO_LARGE before
 * anything is enqueued.  Each call first scans the whole table (count and
 * latest call number), so its cost grows with the capacity.
 * The first call on a device resolves the array's device address with
 * cudaGetSymbolAddress (once per device, on the calling thread's current
 * device); make that first call before any stream capture.
 * All calls share the one array and it keeps the last call's contents: calls
 * whose GPU work overlaps (other streams, other threads, the same device)
 * race on it and must be serialised by the caller.  A table written by this
 * entry point must not be written afterwards through pk_store of a context
 * (their call numbers are not coordinated). */
#define PK_NOALLOC_MAX_ENTRIES (1u << 18)
int pk_store_noalloc(const pk_config *cfg, const uint8_t *keys_dev, const uint32_t *slots_dev, uint64_t n,
                     const int64_t *key_off_dev, const int32_t *hit_chunks_dev, uint32_t R,
                     int32_t *result_dev, uint32_t *slot_out_dev, int32_t *status_dev, pk_stream stream);

/* Host, synchronous.  Number of entries in the table (device counter read
 * after synchronising `stream`). */
int pk_entries(pk_ctx *ctx, uint64_t *count, pk_stream stream);

/* Static description of a status code. */
const char *pk_strerror(int code);

#ifdef __cplusplus
}
#endif

#endif /* PK_H_ */
