// pk_table.cu -- GPU-resident key table: lookup and store kernels (sm_103a).
//
// The shared store of the paper (Sec. 2.1) reduced to its key index: an
// open-addressing table of 2^b entries of 32 bytes (one DRAM sector each),
// keyed by the first 16 bytes of k_i (the 128-bit digest of Sec. 5.3) and
// holding the uint32 slot of the chunk's cached state.  Home position =
// (first 8 key bytes read as a little-endian integer) mod 2^b; linear probing
// with wrap-around; the all-zero key marks an empty entry.  At most
// capacity - 1 entries are ever stored, so every probe meets an empty entry;
// every probe loop is additionally bounded by max_probe.
//
// Lookup (Sec. 2.1: on a local miss the connector queries the store) reads
// the table only.  Store ("a miss computes and writes new state") inserts
// missing keys with a 128-bit compare-and-swap on the key; every entry of the
// call holding a new key bids for it with a 64-bit atomicMax on the entry's
// slot/owner word, so that the lowest entry index's slot is bound, and a
// second kernel reports each entry's outcome: the result equals processing
// the entries one at a time in order.
#include <cuda_runtime.h>

#include "pk_device.cuh"
#include "pk_internal.h"

#include <mutex>

namespace {

using pk::set_status;

__device__ __forceinline__ bool is_zero(const uint4 &v) { return (v.x | v.y | v.z | v.w) == 0u; }
__device__ __forceinline__ bool same(const uint4 &a, const uint4 &b) {
    return ((a.x ^ b.x) | (a.y ^ b.y) | (a.z ^ b.z) | (a.w ^ b.w)) == 0u;
}
__device__ __forceinline__ uint64_t home_of(const uint4 &k) {
    return ((uint64_t)k.y << 32) | k.x;  // bytes 0..7, little-endian
}

// Reads of table entries that other warps of the same kernel may be claiming:
// L2 reads (no L1 copy), issued each time they are asked for.  They only
// guide the probe: every decision that could race is taken by a CAS, and a
// torn read is re-read atomically (examine).
__device__ __forceinline__ uint4 ld_l2_v4(const uint32_t *p) {
    uint4 v;
    asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}
__device__ __forceinline__ unsigned long long ld_volatile_u64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.volatile.global.u64 %0, [%1];" : "=l"(v) : "l"(p));
    return v;
}

// Cooperative probing.  A warp probes the keys of its lanes together.  In
// each round the m keys still undecided are spread over the 32 lanes,
// G = 2^floor(log2(32/m)) lanes per key, and lane j of a key's group loads
// the j-th window of the key's remaining probe sequence: kWin consecutive
// entries (one aligned 128-byte line).  One ballot then finds, in sequence
// order, the first entry that decides the key (its own key, or an empty
// entry).  With a full warp of keys every lane reads one window per round,
// as a lane-per-key probe would; a key whose sequence runs long is joined by
// the lanes whose keys are done, so the warp no longer waits one round trip
// per window for its slowest key.  The entries examined and the decision
// are those of plain linear probing, home, home+1, ...; only the number of
// windows loaded at once differs.
constexpr uint32_t kWin = 4;
constexpr uint32_t kFull = 0xffffffffu;

__device__ __forceinline__ uint32_t lanemask_lt() {
    uint32_t m;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

// Position of the set bit of rank n (0-based, from bit 0) of mask; n < popc(mask).
__device__ __forceinline__ uint32_t nth_set_bit(uint32_t mask, uint32_t n) {
    uint32_t pos = 0;
#pragma unroll
    for (uint32_t s = 16; s >= 1; s >>= 1) {
        const uint32_t low = __popc(mask & ((1u << s) - 1u));
        if (n >= low) {
            n -= low;
            mask >>= s;
            pos += s;
        }
    }
    return pos;
}

__device__ __forceinline__ uint4 shfl4(const uint4 &v, uint32_t src) {
    return make_uint4(__shfl_sync(kFull, v.x, src), __shfl_sync(kFull, v.y, src), __shfl_sync(kFull, v.z, src),
                      __shfl_sync(kFull, v.w, src));
}

// 16-byte load at L2 (coherent: see pk_device.cuh), kept in program order
// (prefetch of the next keys).
__device__ __forceinline__ uint4 ld_cg_v4(const void *p) {
    uint4 v;
    asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// This lane's roles in one round, given the mask P of lanes whose key is
// still undecided.
struct Round {
    uint32_t G;          // lanes per undecided key (power of two)
    uint32_t j;          // worker role: window index within its group
    uint32_t owner;      // worker role: lane holding the key it works on
    bool work;           // worker role: has a key to work on
    uint32_t work_mask;  // lanes of the group it works in
    uint32_t own_mask;   // owner role: lanes working on its own key
};

__device__ __forceinline__ Round plan_round(uint32_t P, uint32_t lane) {
    Round r;
    const uint32_t m = __popc(P);  // >= 1
    const uint32_t lg = 31 - __clz(32u / m);
    r.G = 1u << lg;
    const uint32_t gm = lg == 5 ? kFull : (1u << r.G) - 1u;
    const uint32_t q = lane >> lg;
    r.j = lane & (r.G - 1);
    r.work = q < m;
    r.owner = r.work ? nth_set_bit(P, q) : lane;
    r.work_mask = gm << (q << lg);
    const uint32_t qo = __popc(P & lanemask_lt());
    r.own_mask = ((P >> lane) & 1u) ? gm << (qo << lg) : 0u;
    return r;
}

// Window geometry of a probe position: the aligned window holding it and
// the offset of the position in it.
__device__ __forceinline__ uint32_t window_size(uint64_t mask) { return mask + 1 < kWin ? (uint32_t)(mask + 1) : kWin; }

// A lane's key while it is being probed (owner role).
struct ProbeKey {
    uint4 key;
    uint64_t e;       // entry index of the key in the caller's arrays
    uint64_t pos;     // next table position of its probe sequence
    uint32_t probed;  // entries of the sequence examined so far
    uint32_t slot;    // store: the slot to bind if the key is inserted
    bool pending;     // not decided yet
    bool may_claim;   // lookup-and-store: the key may be inserted (its slot is valid)
};

__device__ __forceinline__ void probe_start(ProbeKey &s, const uint4 &key, uint64_t e, uint64_t mask,
                                            uint32_t slot = 0, bool may_claim = true) {
    s.key = key;
    s.e = e;
    s.slot = slot;
    s.pos = home_of(key) & mask;
    s.probed = 0;
    s.pending = true;
    s.may_claim = may_claim;
}

// Owner role after a round in which no lane of its group found a deciding
// entry: the key's sequence continues after the group's G windows.
__device__ __forceinline__ void skip_windows(ProbeKey &s, uint32_t G, uint32_t win, uint64_t mask) {
    const uint64_t b0 = s.pos & ~(uint64_t)(win - 1);
    s.probed += G * win - (uint32_t)(s.pos - b0);
    s.pos = (b0 + (uint64_t)G * win) & mask;
}

// ---------------------------------------------------------------------------
// Lookup: one round over the undecided keys P of the warp.  Returns true in
// the lanes whose key was decided in this round, with its slot (PK_NO_SLOT
// if absent) and `limit` set if its sequence reached max_probe.
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool lookup_round(const pk_entry *table, uint64_t mask, uint32_t max_probe,
                                             uint32_t P, ProbeKey &s, uint32_t &slot, bool &limit) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t win = window_size(mask);
    // With every lane's key undecided (the common case while a request has
    // keys left) each lane probes its own key and nothing is exchanged.
    const bool full = P == kFull;
    const Round rd = full ? Round{1, 0, lane, true, 1u << lane, 1u << lane} : plan_round(P, lane);
    const uint4 k = full ? s.key : shfl4(s.key, rd.owner);
    const uint64_t wpos = full ? s.pos : __shfl_sync(kFull, s.pos, rd.owner);
    const uint32_t wprobed = full ? s.probed : __shfl_sync(kFull, s.probed, rd.owner);
    const uint64_t base0 = wpos & ~(uint64_t)(win - 1);
    const uint32_t j0 = (uint32_t)(wpos - base0);
    const uint64_t wb = (base0 + (uint64_t)rd.j * win) & mask;
    int cand = -1;
    bool match = false;
    if (rd.work) {
        const pk_entry *grp = table + wb;
        uint4 v[kWin];
#pragma unroll
        for (uint32_t u = 0; u < kWin; ++u) {  // entries before the sequence start are not read
            v[u] = make_uint4(0, 0, 0, 0);
            if (u < win && (rd.j > 0 || u >= j0)) v[u] = __ldcg(reinterpret_cast<const uint4 *>(grp[u].k));
        }
#pragma unroll
        for (uint32_t u = 0; u < kWin; ++u) {
            const bool in_seq = u < win && (rd.j > 0 || u >= j0) && wprobed + (rd.j * win + u - j0) < max_probe;
            if (in_seq && cand < 0) {
                if (same(v[u], k)) {
                    cand = (int)u;
                    match = true;
                } else if (is_zero(v[u])) {
                    cand = (int)u;
                }
            }
        }
    }
    const uint32_t B = __ballot_sync(kFull, cand >= 0);
    const bool decider = cand >= 0 && (B & rd.work_mask & lanemask_lt()) == 0;
    uint32_t dslot = PK_NO_SLOT;
    if (decider && match) dslot = __ldcg(&table[wb + (uint32_t)cand].slot);
    const uint32_t ob = B & rd.own_mask;
    const uint32_t got = full ? dslot : __shfl_sync(kFull, dslot, ob ? __ffs(ob) - 1 : lane);
    if (!s.pending) return false;
    if (ob) {
        slot = got;
        limit = false;
        s.pending = false;
        return true;
    }
    skip_windows(s, rd.G, win, mask);
    if (s.probed >= max_probe) {
        slot = PK_NO_SLOT;
        limit = true;
        s.pending = false;
        return true;
    }
    return false;
}

// One warp per request: every key's slot, and h_r = index of the first miss.
// A lane whose key is decided takes the request's next key, from a register
// buffer holding the next 32 keys (loaded one refill ahead), so the warp
// keeps 32 keys in flight until the request's last keys.
__global__ void __launch_bounds__(256, 4)
k_lookup_req(const pk_entry *table, uint64_t mask, uint32_t max_probe,
             const uint8_t *keys, const int64_t *key_off, uint32_t R,
             uint64_t key_capacity, uint32_t *slots, int32_t *hit, int32_t *status) {
    pk::pdl_wait(table, keys, key_off, slots, hit, status);
    const uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t lane = threadIdx.x & 31;
    if (r >= R) return;  // uniform per warp
    const int64_t a = __ldcg(key_off + r);
    int64_t b = __ldcg(key_off + r + 1);
    if ((uint64_t)b > key_capacity) b = (int64_t)key_capacity;
    uint32_t first_miss = 0xffffffffu;  // lowest missing index (relative to a) seen by this lane
    bool limit = false;
    ProbeKey s;
    s.pending = false;
    bool busy = false;  // holds a key (pending)
    int64_t cursor = a;
    uint4 buf = make_uint4(0, 0, 0, 0);  // key of index cursor + lane
    if (a + lane < b) buf = ld_cg_v4(keys + 32 * (a + lane));
    for (;;) {
        const uint32_t F = __ballot_sync(kFull, !busy);
        if (F) {  // free lanes take the next keys, in lane order
            const uint32_t rank = __popc(F & lanemask_lt());
            const uint4 kin = shfl4(buf, rank);
            if (!busy && cursor + rank < b) {
                const int64_t e = cursor + rank;
                if (is_zero(kin)) {  // the empty marker is never stored
                    slots[e] = PK_NO_SLOT;
                    first_miss = min(first_miss, (uint32_t)(e - a));
                } else {
                    probe_start(s, kin, (uint64_t)e, mask);
                    busy = true;
                }
            }
            const uint32_t nF = __popc(F);
            buf = shfl4(buf, (lane + nF) & 31);
            cursor += nF;
            if (lane + nF >= 32 && cursor + lane < b) buf = ld_cg_v4(keys + 32 * (cursor + lane));
        }
        const uint32_t P = __ballot_sync(kFull, busy);
        if (!P) {
            if (cursor >= b) break;
            continue;
        }
        uint32_t slot;
        bool lim;
        if (lookup_round(table, mask, max_probe, P, s, slot, lim)) {
            slots[s.e] = slot;
            if (slot == PK_NO_SLOT) first_miss = min(first_miss, (uint32_t)((int64_t)s.e - a));
            limit |= lim;
            busy = false;
        }
    }
    pk::pdl_launch_dependents();  // main work done: release the successor (see k_chunk_digest)
    const uint32_t h = __reduce_min_sync(kFull, first_miss);
    if (lane == 0) hit[r] = h != 0xffffffffu ? (int32_t)h : (int32_t)(b > a ? b - a : 0);
    if (limit) set_status(status, PK_ERR_PROBE_LIMIT);
}

// One warp per 32 consecutive keys (few long requests): slots only;
// k_first_miss follows.
__global__ void __launch_bounds__(256)
k_lookup(const pk_entry *table, uint64_t mask, uint32_t max_probe,
         const uint8_t *keys, const int64_t *key_off, uint32_t R,
         uint64_t key_capacity, uint32_t *slots, int32_t *status) {
    pk::pdl_wait(table, keys, key_off, slots, status);
    const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t total = R == 0 ? 0 : __ldcg(key_off + R);
    const int64_t end = total < (int64_t)key_capacity ? total : (int64_t)key_capacity;
    if (g - (int64_t)(threadIdx.x & 31) >= end) return;  // uniform per warp
    ProbeKey s;
    s.pending = false;
    uint32_t slot = PK_NO_SLOT;
    bool limit = false;
    if (g < end) {
        const uint4 key = __ldcg(reinterpret_cast<const uint4 *>(keys + 32 * g));
        if (!is_zero(key)) probe_start(s, key, (uint64_t)g, mask);  // the empty marker is never stored
    }
    for (;;) {
        const uint32_t P = __ballot_sync(kFull, s.pending);
        if (!P) break;
        uint32_t sl;
        bool lim;
        if (lookup_round(table, mask, max_probe, P, s, sl, lim)) {
            slot = sl;
            limit = lim;
        }
    }
    pk::pdl_launch_dependents();
    if (g < end) slots[g] = slot;
    if (limit) set_status(status, PK_ERR_PROBE_LIMIT);
}

// One warp per request: h_r = index of the first PK_NO_SLOT among its keys.
__global__ void __launch_bounds__(256)
k_first_miss(const int64_t *key_off, uint32_t R, uint64_t key_capacity,
             const uint32_t *slots, int32_t *hit) {
    pk::pdl_launch_dependents();
    pk::pdl_wait(key_off, slots, hit);
    const uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t lane = threadIdx.x & 31;
    if (r >= R) return;
    const int64_t a = __ldcg(key_off + r);
    int64_t b = __ldcg(key_off + r + 1);
    if ((uint64_t)b > key_capacity) b = (int64_t)key_capacity;
    int64_t h = b > a ? b - a : 0;
    for (int64_t base = a; base < b; base += 32) {
        const int64_t idx = base + lane;
        const bool miss = idx < b && __ldcg(slots + idx) == PK_NO_SLOT;
        const uint32_t ball = __ballot_sync(kFull, miss);
        if (ball) {
            h = base - a + (__ffs(ball) - 1);
            break;
        }
    }
    if (lane == 0) hit[r] = (int32_t)h;
}

// ---------------------------------------------------------------------------
// Store (Sec. 2.1: a miss computes and writes new state), with the outcome of
// processing the entries one at a time in index order and at most
// capacity - 1 entries ever stored.
//
// Claim kernel, for each entry:
//   key inserted by an earlier call (epoch set, not this call's): PRESENT
//   with its slot, final
//   key claimed in this call (by anyone): bid (~index, slot) on the entry's
//   slot/owner word and leave PENDING with the entry position
//   key absent: in claim mode, CAS the key into the first empty entry (then
//   bid, PENDING); in defer mode, leave the entry DEFERRED for the admission
//   pass and write nothing
// The call takes claim mode when the entry count at its start plus its
// entries stays below capacity: the whole call fits, so no key is refused.
// The count is read from a word no kernel of the call changes, so every warp
// takes the same mode.
// Admission pass, by the claim kernel's last CTA to finish: nothing to do
// unless entries were deferred (a call that may not fit: rare, and then one
// CTA's work).  If the deferred entries fit in the room left (capacity - 1 -
// count), all are claimed; otherwise the CTA walks the deferred entries in
// index order, each round letting at most `room` of them claim (so at most
// `room` new keys), until the room is gone; the rest are bids on keys this
// call already claimed, or TABLE_FULL.  That is exactly the sequential rule:
// the first `room` distinct new keys (by lowest index) go in, later ones are
// refused.  (A separate launch for this pass cost about 2.5 us on every
// store call.)
// Finalize kernel: each PENDING entry reads its key's slot/owner word, final
// once every claim is in: the lowest claimant is INSERTED, the others
// PRESENT with its slot.
//
// Context counter words: [0] entries in the table at the start of the call
// (constant while its claim kernel runs, so that every warp takes the same
// mode), [1] requests handed out by a work-taking lookup-and-store, [2]
// entries deferred in this call, [3] keys its claims claimed, [4] keys its
// admission pass claimed, [5] CTAs of the claim kernel done (reset by the
// last); the finalize kernel adds [3] and [4] to [0] and clears [2..4].
// ---------------------------------------------------------------------------
enum Examine { kAdvance, kDone, kClaimedHere };
enum ClaimMode : uint32_t {
    kModeClaim = 0,   // an absent key is claimed
    kModeDefer = 1,   // an absent key is left DEFERRED (table not written)
    kModeRefuse = 2,  // an absent key is refused (TABLE_FULL)
};

// Bid of entry index e (me = ~e) with its slot for a key new in this call:
// the entry's slot/owner word ends at the maximum bid, that of the lowest
// index, carrying that index's slot.
__device__ __forceinline__ void bid(pk_entry *ent, uint32_t me, uint32_t my_slot) {
    atomicMax(reinterpret_cast<unsigned long long *>(&ent->slot), ((unsigned long long)me << 32) | my_slot);
}

// Examine entry `ent` (position pos) whose key was read as `cur`.
// kFused (lookup-and-store): `lslot` receives the slot of a key that was in
// the table when the call started (inserted by an earlier call: epoch set
// and not this call's), else PK_NO_SLOT; a key that may not be inserted
// (!may_claim) ends with PK_ERR_ARG and leaves the table untouched.
// stamps (budget mode, else NULL): the last-use stamp (epoch << 32) | e of
// the key's entry is raised to this entry's when the key was in the table at
// the start of the call, or is inserted by it with a valid slot.
template <bool kFused>
__device__ __forceinline__ Examine examine(pk_entry *ent, uint64_t pos, uint4 cur, const uint4 &key, uint32_t me,
                                           uint32_t my_slot, unsigned long long epoch, uint32_t mode, bool may_claim,
                                           unsigned long long *stamps, int32_t &res, uint32_t &out, uint32_t &lslot) {
    uint4 *kp = reinterpret_cast<uint4 *>(ent->k);
    const unsigned long long my_stamp = (epoch << 32) | (unsigned long long)(uint32_t)~me;
    lslot = PK_NO_SLOT;
#pragma unroll 1
    for (int pass = 0; pass < 2; ++pass) {
        // A vector load racing a concurrent 128-bit CAS may observe a mix of
        // zero and new words.  When every word is zero or equal to ours, take
        // an atomic snapshot: a CAS that swaps our key for itself changes
        // nothing and returns the entry's whole current key.
        if (!same(cur, key) && !is_zero(cur) && (cur.x == 0 || cur.x == key.x) && (cur.y == 0 || cur.y == key.y) &&
            (cur.z == 0 || cur.z == key.z) && (cur.w == 0 || cur.w == key.w))
            cur = atomicCAS(kp, key, key);
        if (same(cur, key)) {
            const uint4 m = ld_l2_v4(&ent->slot);  // slot, owner, epoch in one read
            const unsigned long long ep = ((unsigned long long)m.w << 32) | m.z;
            if (ep != 0ull && ep != epoch) {  // inserted by an earlier call
                const uint32_t sl = m.x;
                if (kFused) lslot = sl;
                res = (!kFused || may_claim) ? PK_STORE_PRESENT : PK_ERR_ARG;
                out = (!kFused || may_claim) ? sl : PK_NO_SLOT;
                if (stamps) atomicMax(stamps + pos, my_stamp);
            } else if (!kFused || may_claim) {  // claimed during this call
                bid(ent, me, my_slot);
                res = PK_STORE_PENDING;
                out = (uint32_t)pos;
                if (stamps) atomicMax(stamps + pos, my_stamp);
            } else {
                res = PK_ERR_ARG;
                out = PK_NO_SLOT;
            }
            return kDone;
        }
        if (!is_zero(cur)) return kAdvance;  // a different key holds this entry
        if (kFused && !may_claim) {          // absent; not to be inserted
            res = PK_ERR_ARG;
            out = PK_NO_SLOT;
            return kDone;
        }
        if (mode != kModeClaim) {  // absent: left to the admission pass, or refused
            res = mode == kModeDefer ? PK_STORE_DEFERRED : PK_ERR_TABLE_FULL;
            out = PK_NO_SLOT;
            return kDone;
        }
        const uint4 old = atomicCAS(kp, make_uint4(0, 0, 0, 0), key);
        if (is_zero(old)) {  // claimed
            *(volatile unsigned long long *)&ent->epoch = epoch;
            bid(ent, me, my_slot);
            if (stamps) atomicMax(stamps + pos, my_stamp);
            res = PK_STORE_PENDING;
            out = (uint32_t)pos;
            return kClaimedHere;  // counted once per block at the end
        }
        cur = old;  // examine the winner's key
    }
    return kAdvance;
}

// An entry read as v can decide key k: it is empty, holds k, or is a torn
// read of k being written (every word zero or k's).
__device__ __forceinline__ bool may_decide(const uint4 &v, const uint4 &k) {
    return (v.x == 0 || v.x == k.x) && (v.y == 0 || v.y == k.y) && (v.z == 0 || v.z == k.z) &&
           (v.w == 0 || v.w == k.w);
}

// Where a table is shared by the claims of one store call.
struct ClaimCtx {
    pk_entry *table;
    uint64_t mask;
    uint32_t max_probe;
    unsigned long long epoch;
    uint32_t mode;               // ClaimMode: what happens to an absent key
    unsigned long long *stamps;  // budget mode: last-use stamp per entry, else NULL
};

// Mode of a claim kernel's warp: claim when the entry count at the start of
// the call plus the call's entries stays below capacity (the whole call
// fits), else defer.
__device__ __forceinline__ uint32_t claim_mode(const unsigned long long *counter, uint64_t n, uint64_t capacity) {
    unsigned long long cnt = 0;
    if ((threadIdx.x & 31) == 0) cnt = ld_volatile_u64(counter);
    return __shfl_sync(kFull, cnt, 0) + n < capacity ? kModeClaim : kModeDefer;
}

// Insert-if-absent: one round over the undecided keys P of the warp.
// Returns true in the lanes whose key was decided in this round, with its
// result code and output; `claims` counts the claims this lane made as
// decider (for any key of the warp).
// kFused: also `lslot`, the key's slot if it was in the table when the call
// started (else PK_NO_SLOT), and keys with !may_claim are looked up only.
template <bool kFused>
__device__ __forceinline__ bool claim_round(const ClaimCtx &c, uint32_t P, ProbeKey &s, int32_t &res,
                                            uint32_t &out, uint32_t &lslot, uint32_t &claims) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t win = window_size(c.mask);
    const bool full = P == kFull;  // as in lookup_round
    const Round rd = full ? Round{1, 0, lane, true, 1u << lane, 1u << lane} : plan_round(P, lane);
    const uint4 k = full ? s.key : shfl4(s.key, rd.owner);
    const uint64_t wpos = full ? s.pos : __shfl_sync(kFull, s.pos, rd.owner);
    const uint32_t wprobed = full ? s.probed : __shfl_sync(kFull, s.probed, rd.owner);
    const uint64_t we = full ? s.e : __shfl_sync(kFull, s.e, rd.owner);
    const bool wmay = !kFused || (full ? s.may_claim : __shfl_sync(kFull, (int)s.may_claim, rd.owner) != 0);
    const uint32_t wslot = full ? s.slot : __shfl_sync(kFull, s.slot, rd.owner);
    const uint64_t base0 = wpos & ~(uint64_t)(win - 1);
    const uint32_t j0 = (uint32_t)(wpos - base0);
    const uint64_t wb = (base0 + (uint64_t)rd.j * win) & c.mask;
    int cand = -1;
    uint32_t cseq = 0;
    uint4 cv = make_uint4(0, 0, 0, 0);
    if (rd.work) {
        pk_entry *grp = c.table + wb;
        uint4 v[kWin];
#pragma unroll
        for (uint32_t u = 0; u < kWin; ++u) {  // entries before the sequence start are not read
            v[u] = make_uint4(0, 0, 0, 0);
            if (u < win && (rd.j > 0 || u >= j0)) v[u] = ld_l2_v4(grp[u].k);
        }
#pragma unroll
        for (uint32_t u = 0; u < kWin; ++u) {
            const uint32_t seq = rd.j * win + u - j0;
            const bool in_seq = u < win && (rd.j > 0 || u >= j0) && wprobed + seq < c.max_probe;
            if (in_seq && cand < 0 && may_decide(v[u], k)) {
                cand = (int)u;
                cseq = seq;
                cv = v[u];
            }
        }
    }
    const uint32_t B = __ballot_sync(kFull, cand >= 0);
    const bool decider = cand >= 0 && (B & rd.work_mask & lanemask_lt()) == 0;
    int32_t dres = PK_ERR_PROBE_LIMIT;
    uint32_t dout = PK_NO_SLOT, dls = PK_NO_SLOT;
    bool dadv = false;
    uint64_t dnext = 0;
    uint32_t dprobed = 0;
    if (decider) {
        const uint64_t epos = wb + (uint32_t)cand;
        const Examine x = examine<kFused>(c.table + epos, epos, cv, k, ~(uint32_t)we, wslot, c.epoch, c.mode, wmay,
                                          c.stamps, dres, dout, dls);
        if (x == kClaimedHere) ++claims;
        if (x == kAdvance) {  // lost the entry to a different key: continue after it
            dadv = true;
            dnext = (epos + 1) & c.mask;
            dprobed = wprobed + cseq + 1;
        }
    }
    const uint32_t ob = B & rd.own_mask;
    int32_t g_res = dres;
    uint32_t g_out = dout, g_probed = dprobed, g_ls = dls;
    bool g_adv = dadv;
    uint64_t g_next = dnext;
    if (!full) {
        const uint32_t src = ob ? __ffs(ob) - 1 : lane;
        g_res = __shfl_sync(kFull, dres, src);
        g_out = __shfl_sync(kFull, dout, src);
        if (kFused) g_ls = __shfl_sync(kFull, dls, src);
        g_adv = __shfl_sync(kFull, (int)dadv, src) != 0;
        g_next = __shfl_sync(kFull, dnext, src);
        g_probed = __shfl_sync(kFull, dprobed, src);
    }
    if (!s.pending) return false;
    if (ob && !g_adv) {
        res = g_res;
        out = g_out;
        lslot = g_ls;
        s.pending = false;
        return true;
    }
    if (ob) {
        s.pos = g_next;
        s.probed = g_probed;
    } else {
        skip_windows(s, rd.G, win, c.mask);
    }
    if (s.probed >= c.max_probe) {
        res = PK_ERR_PROBE_LIMIT;
        out = PK_NO_SLOT;
        lslot = PK_NO_SLOT;
        s.pending = false;
        return true;
    }
    return false;
}

// Insert-if-absent (kFused: lookup-and-store) of at most one key per lane,
// all lanes together.
template <bool kFused>
__device__ __forceinline__ void warp_claim(const ClaimCtx &c, ProbeKey &s, int32_t &res, uint32_t &out,
                                           uint32_t &lslot, uint32_t &claims) {
    for (;;) {
        const uint32_t P = __ballot_sync(kFull, s.pending);
        if (!P) break;
        claim_round<kFused>(c, P, s, res, out, lslot, claims);
    }
}

// Argument checks of one entry before it is claimed: a zero key is the
// empty marker; PK_NO_SLOT is not a storable slot.
__device__ __forceinline__ bool claimable(const uint4 &key, uint32_t slot, int32_t &res) {
    if (is_zero(key)) {
        res = PK_ERR_RESERVED_KEY;
        return false;
    }
    if (slot == PK_NO_SLOT) {
        res = PK_ERR_ARG;
        return false;
    }
    return true;
}

// Whether entry e lies in the store range of its request, [key_off[r] + h_r,
// key_off[r+1]) (range mode; warp-collective).
__device__ __forceinline__ bool in_store_range(const int64_t *key_off, const int32_t *hit,
                                               uint32_t R, uint64_t n, uint64_t e) {
    const uint64_t e0 = e - (threadIdx.x & 31);
    const int64_t total = R > 0 ? __ldcg(key_off + R) : 0;
    bool in_range = false;
    if (e0 < n && (int64_t)e0 < total) {
        const uint32_t r = pk::lane_request(key_off, R, (int64_t)e0, total, (int64_t)e);
        if ((int64_t)e < total) {
            const int64_t h = __ldcg(hit + r);
            in_range = (int64_t)e - __ldcg(key_off + r) >= (h > 0 ? h : 0);
        }
    }
    return in_range;
}

// Adds the warp's claims and deferred entries to the block totals, then the
// block totals to counter[3] (claims) and counter[2] (deferred): one atomic
// per block and word (same-address atomics serialise in L2).
__device__ __forceinline__ void count_claims(unsigned long long *block_sums, uint32_t claims, uint32_t deferred,
                                             unsigned long long *counter) {
    const uint32_t w = __reduce_add_sync(kFull, claims);
    const uint32_t d = __reduce_add_sync(kFull, deferred);
    if ((threadIdx.x & 31) == 0 && w) atomicAdd_block(block_sums, (unsigned long long)w);
    if ((threadIdx.x & 31) == 0 && d) atomicAdd_block(block_sums + 1, (unsigned long long)d);
    __syncthreads();
    if (threadIdx.x == 0 && block_sums[0]) atomicAdd(counter + 3, block_sums[0]);
    if (threadIdx.x == 0 && block_sums[1]) atomicAdd(counter + 2, block_sums[1]);
}

// Result of a deferred entry decided by the admission pass.  pos_out: where a
// PENDING entry's table position goes (slot_out for a context; the
// allocation-free store keeps positions apart and writes PK_NO_SLOT to
// slot_out).
__device__ __forceinline__ void admit_write(uint64_t e, int32_t res, uint32_t out, int32_t *result,
                                            uint32_t *slot_out, uint32_t *pos_out, int32_t *status) {
    result[e] = res;
    if (res == PK_STORE_PENDING && pos_out != slot_out) {
        pos_out[e] = out;
        slot_out[e] = PK_NO_SLOT;
    } else {
        slot_out[e] = out;
    }
    if (res < 0) set_status(status, res);
}

// Store, admission pass (see the store comment above), run by one CTA: the
// last CTA of the claim kernel to finish.  The call's entries are [0, n), or
// [0, min(n, key_off[R])) in range and lookup-and-store mode; counter[0] +
// counter[3] is the entry count after the claims, counter[2] the number of
// DEFERRED entries; keys claimed here are added to counter[4].  Within the
// call the entry count can only reach capacity - 1: the claim kernel claims
// only when the whole call fits, and here at most `room` keys are claimed.
// Out of line: the claim kernels' registers stay those of their main loops.
__device__ __noinline__ void store_admit(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
                                            unsigned long long *counter, unsigned long long epoch,
                                            unsigned long long *stamps, const uint8_t *keys, const uint32_t *slots,
                                            uint64_t n, const int64_t *key_off, uint32_t R, int32_t *result,
                                            uint32_t *slot_out, uint32_t *pos_out, int32_t *status) {
    __shared__ uint32_t s_warp[8];
    __shared__ unsigned long long s_claims;
    const unsigned long long deferred = __ldcg(counter + 2);
    if (deferred == 0) return;  // every key was decided by the claim kernel
    const unsigned long long count = __ldcg(counter) + __ldcg(counter + 3);
    const unsigned long long room = count + 1 < capacity ? capacity - 1 - count : 0ull;
    uint64_t end = n;
    if (key_off) {
        const int64_t t = R ? __ldcg(key_off + R) : 0;
        if (t < (int64_t)end) end = t > 0 ? (uint64_t)t : 0;
    }
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (deferred <= room) {
        // At most `deferred` distinct keys: all fit.  Claimed by all warps of the CTA at once.
        const ClaimCtx c{table, mask, max_probe, epoch, kModeClaim, stamps};
        uint32_t claims = 0;
        if (threadIdx.x == 0) s_claims = 0;
        __syncthreads();
        for (uint64_t base = 32 * warp; base < end; base += blockDim.x) {  // uniform per warp
            const uint64_t e = base + lane;
            ProbeKey s;
            s.pending = false;
            if (e < end && __ldcg(result + e) == PK_STORE_DEFERRED)
                probe_start(s, ld_cg_v4(keys + 32 * e), e, mask, __ldcg(slots + e));
            const bool mine = s.pending;
            int32_t res;
            uint32_t out, lslot;
            warp_claim<false>(c, s, res, out, lslot, claims);
            if (mine) admit_write(e, res, out, result, slot_out, pos_out, status);
        }
        const uint32_t wc = __reduce_add_sync(kFull, claims);
        if (lane == 0 && wc) atomicAdd_block(&s_claims, (unsigned long long)wc);
        __syncthreads();
        if (threadIdx.x == 0 && s_claims) atomicAdd(counter + 4, s_claims);
        return;
    }
    // More deferred entries than room: walk them in index order, one tile of
    // blockDim.x at a time.  Each round the first `left` undecided entries of
    // the tile (at most `left` distinct keys) claim or bid; once the room is
    // gone the rest only bid on keys this call claimed, or are refused.  Every
    // round decides at least one entry.
    unsigned long long left = room, admitted = 0;
    for (uint64_t base = 0; base < end; base += blockDim.x) {
        const uint64_t e = base + threadIdx.x;
        bool pend = e < end && __ldcg(result + e) == PK_STORE_DEFERRED;
        const uint4 key = pend ? ld_cg_v4(keys + 32 * e) : make_uint4(0, 0, 0, 0);
        const uint32_t sl = pend ? __ldcg(slots + e) : 0u;
        for (;;) {
            const uint32_t ball = __ballot_sync(kFull, pend);
            if (lane == 0) s_warp[warp] = __popc(ball);
            if (threadIdx.x == 0) s_claims = 0;
            if (__syncthreads_count(pend) == 0) break;  // the tile is decided (uniform)
            uint32_t rank = __popc(ball & lanemask_lt());
            for (uint32_t w = 0; w < warp; ++w) rank += s_warp[w];
            const bool act = pend && (left == 0 || rank < left);
            const ClaimCtx c{table, mask, max_probe, epoch, left == 0 ? kModeRefuse : kModeClaim, stamps};
            ProbeKey s;
            s.pending = false;
            if (act) probe_start(s, key, e, mask, sl);
            uint32_t claims = 0;
            int32_t res;
            uint32_t out, lslot;
            warp_claim<false>(c, s, res, out, lslot, claims);
            if (act) {
                admit_write(e, res, out, result, slot_out, pos_out, status);
                pend = false;
            }
            const uint32_t wc = __reduce_add_sync(kFull, claims);
            if (lane == 0 && wc) atomicAdd_block(&s_claims, (unsigned long long)wc);
            __syncthreads();
            left -= s_claims;  // <= left: at most `left` entries claimed
            admitted += s_claims;
            __syncthreads();  // s_warp and s_claims are rewritten next round
        }
    }
    if (threadIdx.x == 0 && admitted) atomicAdd(counter + 4, admitted);
}

// End of a claim kernel: the last CTA to finish (every CTA counts itself on
// counter[5] after a fence) runs the admission pass when the call deferred
// entries, and resets counter[5] for the next call.  Every CTA of the grid
// must call it.
__device__ __forceinline__ void admit_if_last(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
                                              unsigned long long *counter, unsigned long long epoch,
                                              unsigned long long *stamps, const uint8_t *keys, const uint32_t *slots,
                                              uint64_t n, const int64_t *key_off, uint32_t R, int32_t *result,
                                              uint32_t *slot_out, uint32_t *pos_out, int32_t *status) {
    __shared__ int s_last;
    __threadfence();  // this CTA's results and counts are visible to the GPU before it counts itself
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(counter + 5, 1ull) == (unsigned long long)gridDim.x - 1ull;
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (threadIdx.x == 0) counter[5] = 0;
    if (__ldcg(counter + 2) == 0) return;  // nothing deferred: the claim kernel decided every entry
    store_admit(table, mask, max_probe, capacity, counter, epoch, stamps, keys, slots, n, key_off, R, result,
                slot_out, pos_out, status);
}

// List mode, or range mode for few long requests: one warp per 32
// consecutive entries.
__global__ void __launch_bounds__(256, 4)
k_store_claim(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
              unsigned long long *counter, unsigned long long epoch, unsigned long long *stamps, const uint8_t *keys,
              const uint32_t *slots, uint64_t n, const int64_t *key_off,
              const int32_t *hit, uint32_t R, int32_t *result,
              uint32_t *slot_out, int32_t *status) {
    __shared__ unsigned long long block_sums[2];
    if (threadIdx.x < 2) block_sums[threadIdx.x] = 0;
    __syncthreads();
    pk::pdl_wait(table, counter, keys, slots, key_off, hit, result, slot_out, status);
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    bool active = e < n;
    if (key_off) active = in_store_range(key_off, hit, R, n, e) && active;
    const ClaimCtx c{table, mask, max_probe, epoch, claim_mode(counter, n, capacity), stamps};
    int32_t res = PK_STORE_SKIPPED;
    uint32_t out = PK_NO_SLOT;
    ProbeKey s;
    s.pending = false;
    if (active) {
        const uint4 key = __ldcg(reinterpret_cast<const uint4 *>(keys + 32 * e));
        const uint32_t sl = slots[e];
        if (claimable(key, sl, res)) probe_start(s, key, e, mask, sl);
    }
    uint32_t claims = 0, lslot;
    warp_claim<false>(c, s, res, out, lslot, claims);
    if (e < n) {
        result[e] = res;
        slot_out[e] = out;
        if (res < 0) set_status(status, res);
    }
    pk::pdl_launch_dependents();
    count_claims(block_sums, claims, e < n && res == PK_STORE_DEFERRED, counter);
    admit_if_last(table, mask, max_probe, capacity, counter, epoch, stamps, keys, slots, n, key_off, R, result, slot_out,
                  slot_out, status);
}

// Range mode for many short requests: one warp per request, no search.
// Writes every entry of [key_off[r], key_off[r+1]); entries past key_off[R]
// are marked by the finalize kernel.
__global__ void __launch_bounds__(256, 3)
k_store_claim_req(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
                  unsigned long long *counter, unsigned long long epoch, unsigned long long *stamps, const uint8_t *keys,
                  const uint32_t *slots, uint64_t n, const int64_t *key_off,
                  const int32_t *hit, uint32_t R, int32_t *result,
                  uint32_t *slot_out, int32_t *status) {
    __shared__ unsigned long long block_sums[2];
    if (threadIdx.x < 2) block_sums[threadIdx.x] = 0;
    __syncthreads();
    pk::pdl_wait(table, counter, keys, slots, key_off, hit, result, slot_out, status);
    const uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t lane = threadIdx.x & 31;
    int64_t a = 0, b = 0, first = 0;
    if (r < R) {  // uniform per warp
        a = __ldcg(key_off + r);
        b = __ldcg(key_off + r + 1);
        if ((uint64_t)b > n) b = (int64_t)n;
        const int64_t h0 = __ldcg(hit + r);
        first = a + (h0 > 0 ? h0 : 0);
    }
    const ClaimCtx c{table, mask, max_probe, epoch, claim_mode(counter, n, capacity), stamps};
    uint32_t claims = 0, deferred = 0;
    for (int64_t x = a + lane; x < first && x < b; x += 32) {  // below h_r: not stored
        result[x] = PK_STORE_SKIPPED;
        slot_out[x] = PK_NO_SLOT;
    }
    // The store range [first, b): a lane whose key is decided takes the next
    // one from a register buffer of the next 32 keys and slots (as in
    // k_lookup_req).
    ProbeKey s;
    s.pending = false;
    int64_t cursor = first;
    uint4 buf = make_uint4(0, 0, 0, 0);  // key and slot of index cursor + lane
    uint32_t buf_slot = 0;
    if (first + lane < b) {
        buf = ld_cg_v4(keys + 32 * (first + lane));
        buf_slot = __ldcg(slots + first + lane);
    }
    for (;;) {
        const uint32_t F = __ballot_sync(kFull, !s.pending);
        if (F) {  // free lanes take the next keys, in lane order
            const uint32_t rank = __popc(F & lanemask_lt());
            const uint4 kin = shfl4(buf, rank);
            const uint32_t sin = __shfl_sync(kFull, buf_slot, rank);
            if (!s.pending && cursor + rank < b) {
                const int64_t e = cursor + rank;
                int32_t res;
                if (claimable(kin, sin, res)) {
                    probe_start(s, kin, (uint64_t)e, mask, sin);
                } else {
                    result[e] = res;
                    slot_out[e] = PK_NO_SLOT;
                    set_status(status, res);
                }
            }
            const uint32_t nF = __popc(F);
            buf = shfl4(buf, (lane + nF) & 31);
            buf_slot = __shfl_sync(kFull, buf_slot, (lane + nF) & 31);
            cursor += nF;
            if (lane + nF >= 32 && cursor + lane < b) {
                buf = ld_cg_v4(keys + 32 * (cursor + lane));
                buf_slot = __ldcg(slots + cursor + lane);
            }
        }
        const uint32_t P = __ballot_sync(kFull, s.pending);
        if (!P) {
            if (cursor >= b) break;
            continue;
        }
        int32_t res;
        uint32_t out, lslot;
        if (claim_round<false>(c, P, s, res, out, lslot, claims)) {
            result[s.e] = res;
            slot_out[s.e] = out;
            if (res < 0) set_status(status, res);
            deferred += res == PK_STORE_DEFERRED;
        }
    }
    pk::pdl_launch_dependents();
    count_claims(block_sums, claims, deferred, counter);
    admit_if_last(table, mask, max_probe, capacity, counter, epoch, stamps, keys, slots, n, key_off, R, result, slot_out,
                  slot_out, status);
}

// ---------------------------------------------------------------------------
// Lookup and store in one pass (pk_lookup_store).  Every key of the batch is
// inserted if absent, and keys inserted earlier in the same call count as
// absent: a key inserted by an earlier call is a hit (with its slot), any
// other key a miss.  That is the lookup of the table as of the start of the
// call.  h_r is the first miss of request r and every miss lies at or after
// h_r, so the insertions made are exactly those of storing [h_r, n_r) after
// the lookup; the entries below h_r (all hits) are then relabelled
// PK_STORE_SKIPPED.  A key whose slot is PK_NO_SLOT is only looked up and
// ends with PK_ERR_ARG when it lies in the store range.
// ---------------------------------------------------------------------------

// One request r (warp-uniform; r >= R does nothing), refilled from a register
// buffer as k_lookup_req.  `release`: release the finalize launch after the
// probes (the kernel with one request per warp).
__device__ __forceinline__ void lookup_store_request(const ClaimCtx &c, uint64_t r, const uint8_t *keys,
                                                     const uint32_t *new_slots, const int64_t *key_off, uint32_t R,
                                                     uint64_t key_capacity, uint32_t *slots, int32_t *hit,
                                                     int32_t *result, uint32_t *slot_out, int32_t *status,
                                                     uint32_t &claims, uint32_t &deferred, bool release) {
    const uint64_t mask = c.mask;
    const uint32_t lane = threadIdx.x & 31;
    int64_t a = 0, b = 0;
    if (r < R) {  // uniform per warp
        a = __ldcg(key_off + r);
        b = __ldcg(key_off + r + 1);
        if ((uint64_t)b > key_capacity) b = (int64_t)key_capacity;
    }
    uint32_t first_miss = 0xffffffffu;  // lowest miss index (relative to a) seen by this lane
    int64_t arg_hit = -1;               // highest index of a hit whose slot was PK_NO_SLOT
    ProbeKey s;
    s.pending = false;
    int64_t cursor = a;
    uint4 buf = make_uint4(0, 0, 0, 0);  // key and slot of index cursor + lane
    uint32_t buf_slot = 0;
    if (a + lane < b) {
        buf = ld_cg_v4(keys + 32 * (a + lane));
        buf_slot = __ldcg(new_slots + a + lane);
    }
    for (;;) {
        const uint32_t F = __ballot_sync(kFull, !s.pending);
        if (F) {  // free lanes take the next keys, in lane order
            const uint32_t rank = __popc(F & lanemask_lt());
            const uint4 kin = shfl4(buf, rank);
            const uint32_t sin = __shfl_sync(kFull, buf_slot, rank);
            if (!s.pending && cursor + rank < b) {
                const int64_t e = cursor + rank;
                if (is_zero(kin)) {  // the empty marker: never stored, so a miss
                    slots[e] = PK_NO_SLOT;
                    result[e] = PK_ERR_RESERVED_KEY;
                    slot_out[e] = PK_NO_SLOT;
                    set_status(status, PK_ERR_RESERVED_KEY);
                    first_miss = min(first_miss, (uint32_t)(e - a));
                } else {
                    probe_start(s, kin, (uint64_t)e, mask, sin, sin != PK_NO_SLOT);
                }
            }
            const uint32_t nF = __popc(F);
            buf = shfl4(buf, (lane + nF) & 31);
            buf_slot = __shfl_sync(kFull, buf_slot, (lane + nF) & 31);
            cursor += nF;
            if (lane + nF >= 32 && cursor + lane < b) {
                buf = ld_cg_v4(keys + 32 * (cursor + lane));
                buf_slot = __ldcg(new_slots + cursor + lane);
            }
        }
        const uint32_t P = __ballot_sync(kFull, s.pending);
        if (!P) {
            if (cursor >= b) break;
            continue;
        }
        int32_t res;
        uint32_t out, lslot;
        if (claim_round<true>(c, P, s, res, out, lslot, claims)) {
            const int64_t e = (int64_t)s.e;
            slots[e] = lslot;
            result[e] = res;
            slot_out[e] = out;
            deferred += res == PK_STORE_DEFERRED;
            if (lslot == PK_NO_SLOT) {
                first_miss = min(first_miss, (uint32_t)(e - a));
                if (res < 0) set_status(status, res);
            } else if (res < 0) {
                arg_hit = e > arg_hit ? e : arg_hit;
            }
        }
    }
    if (release) pk::pdl_launch_dependents();  // main work done: release the finalize kernel
    const uint32_t hm = __reduce_min_sync(kFull, first_miss);
    const int64_t h = hm != 0xffffffffu ? (int64_t)hm : (b > a ? b - a : 0);
    __syncwarp();
    for (int64_t x = a + lane; x < a + h; x += 32) {  // below h_r: looked up, not stored
        result[x] = PK_STORE_SKIPPED;
        slot_out[x] = PK_NO_SLOT;
    }
    if (r < R && lane == 0) hit[r] = (int32_t)h;
    if (arg_hit >= a + h) set_status(status, PK_ERR_ARG);
}

// Next request for a work-taking warp: tickets[0] counts the requests handed
// out in this call (zeroed before the launch).
__device__ __forceinline__ uint64_t take_request(unsigned long long *tickets) {
    unsigned long long t = 0;
    if ((threadIdx.x & 31) == 0) t = atomicAdd(tickets, 1ull);
    return __shfl_sync(kFull, t, 0);
}

// One warp per request (kTake false: warp w serves request w), or a grid of
// resident CTAs whose warps take requests one at a time until none is left
// (kTake true, for batches of more requests than resident warps: a warp done
// with its request does not wait for the slowest request of its block).
constexpr unsigned kLsBlock = 128;  // 72 registers: 7 CTAs (28 warps) per SM, against 3 CTAs (24 warps) of 256

template <bool kTake>
__global__ void __launch_bounds__(kLsBlock, 7)
k_lookup_store_req(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity,
                   unsigned long long *counter, unsigned long long epoch, unsigned long long *stamps, const uint8_t *keys,
                   const uint32_t *new_slots, const int64_t *key_off, uint32_t R,
                   uint64_t key_capacity, uint32_t *slots, int32_t *hit,
                   int32_t *result, uint32_t *slot_out, int32_t *status, unsigned long long *tickets) {
    __shared__ unsigned long long block_sums[2];
    if (threadIdx.x < 2) block_sums[threadIdx.x] = 0;
    __syncthreads();
    pk::pdl_wait(table, counter, keys, new_slots, key_off, slots, hit, result, slot_out, status, tickets);
    const ClaimCtx c{table, mask, max_probe, epoch, claim_mode(counter, key_capacity, capacity), stamps};
    uint32_t claims = 0, deferred = 0;
    if (kTake) {
        for (uint64_t r = take_request(tickets); r < R; r = take_request(tickets))
            lookup_store_request(c, r, keys, new_slots, key_off, R, key_capacity, slots, hit, result, slot_out,
                                 status, claims, deferred, false);
        pk::pdl_launch_dependents();
    } else {
        const uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
        lookup_store_request(c, r, keys, new_slots, key_off, R, key_capacity, slots, hit, result, slot_out, status,
                             claims, deferred, true);
    }
    count_claims(block_sums, claims, deferred, counter);
    admit_if_last(table, mask, max_probe, capacity, counter, epoch, stamps, keys, new_slots, key_capacity, key_off, R,
                  result, slot_out, slot_out, status);
}

// Few long requests: one warp per 32 consecutive keys; k_lookup_store_tail
// then finds h_r and relabels.
__global__ void __launch_bounds__(256)
k_lookup_store(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity, unsigned long long *counter,
               unsigned long long epoch, unsigned long long *stamps, const uint8_t *keys, const uint32_t *new_slots,
               const int64_t *key_off, uint32_t R, uint64_t key_capacity, uint32_t *slots,
               int32_t *result, uint32_t *slot_out, int32_t *status) {
    __shared__ unsigned long long block_sums[2];
    if (threadIdx.x < 2) block_sums[threadIdx.x] = 0;
    __syncthreads();
    pk::pdl_wait(table, counter, keys, new_slots, key_off, slots, result, slot_out, status);
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t total = R == 0 ? 0 : __ldcg(key_off + R);
    const int64_t end = total < (int64_t)key_capacity ? total : (int64_t)key_capacity;
    const ClaimCtx c{table, mask, max_probe, epoch, claim_mode(counter, key_capacity, capacity), stamps};
    int32_t res = PK_STORE_SKIPPED;
    uint32_t out = PK_NO_SLOT, lslot = PK_NO_SLOT;
    ProbeKey s;
    s.pending = false;
    if (e < end) {
        const uint4 key = __ldcg(reinterpret_cast<const uint4 *>(keys + 32 * e));
        const uint32_t sl = __ldcg(new_slots + e);
        if (is_zero(key))
            res = PK_ERR_RESERVED_KEY;  // the empty marker: never stored, so a miss
        else
            probe_start(s, key, (uint64_t)e, mask, sl, sl != PK_NO_SLOT);
    }
    uint32_t claims = 0;
    warp_claim<true>(c, s, res, out, lslot, claims);
    if (e < end) {
        slots[e] = lslot;
        result[e] = res;
        slot_out[e] = out;
        if (lslot == PK_NO_SLOT && res < 0) set_status(status, res);
    }
    pk::pdl_launch_dependents();
    count_claims(block_sums, claims, e < end && res == PK_STORE_DEFERRED, counter);
    admit_if_last(table, mask, max_probe, capacity, counter, epoch, stamps, keys, new_slots, key_capacity, key_off, R,
                  result, slot_out, slot_out, status);
}

// One warp per request: h_r = the first miss (slot PK_NO_SLOT), entries below
// it relabelled PK_STORE_SKIPPED, and PK_ERR_ARG reported for a hit at or
// after h_r whose slot was PK_NO_SLOT.
__global__ void __launch_bounds__(256)
k_lookup_store_tail(const int64_t *key_off, uint32_t R, uint64_t key_capacity,
                    const uint32_t *slots, int32_t *hit, int32_t *result,
                    uint32_t *slot_out, int32_t *status) {
    pk::pdl_launch_dependents();
    pk::pdl_wait(key_off, slots, hit, result, slot_out, status);
    const uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t lane = threadIdx.x & 31;
    if (r >= R) return;
    const int64_t a = __ldcg(key_off + r);
    int64_t b = __ldcg(key_off + r + 1);
    if ((uint64_t)b > key_capacity) b = (int64_t)key_capacity;
    int64_t h = b > a ? b - a : 0;
    bool arg = false;
    for (int64_t base = a; base < b; base += 32) {
        const int64_t x = base + lane;
        const bool in = x < b;
        const uint32_t sl = in ? slots[x] : 0u;
        const uint32_t ball = __ballot_sync(kFull, in && sl == PK_NO_SLOT);
        const int64_t hb = ball ? base - a + (__ffs(ball) - 1) : INT64_MAX;
        if (h == b - a && hb < h) h = hb;  // first miss found in this group
        if (in && x >= a + h) arg |= sl != PK_NO_SLOT && result[x] == PK_ERR_ARG;
    }
    for (int64_t x = a + lane; x < a + h; x += 32) {
        result[x] = PK_STORE_SKIPPED;
        slot_out[x] = PK_NO_SLOT;
    }
    if (lane == 0) hit[r] = (int32_t)h;
    if (arg) set_status(status, PK_ERR_ARG);
}

// Store, last kernel: each PENDING entry reads its key's slot/owner word,
// final once every claim is in: the lowest claimant is INSERTED, the others
// PRESENT with its slot.  In range mode, entries past key_off[R] (not keys
// of this batch) are skipped.  The call's claims are added to the entry
// count, and its counter words [2..4] cleared.
__global__ void __launch_bounds__(256)
k_store_finalize(const pk_entry *table, uint64_t n, const int64_t *key_off, uint32_t R,
                 int32_t *result, uint32_t *slot_out, unsigned long long *counter) {
    pk::pdl_launch_dependents();
    pk::pdl_wait(table, key_off, result, slot_out, counter);
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e == 0) {
        const unsigned long long c2 = __ldcg(counter + 2), c3 = __ldcg(counter + 3), c4 = __ldcg(counter + 4);
        if (c3 | c4) counter[0] += c3 + c4;
        if (c2 | c3 | c4) {
            counter[2] = 0;
            counter[3] = 0;
            counter[4] = 0;
        }
    }
    if (e >= n) return;
    if (key_off && (int64_t)e >= (R > 0 ? __ldcg(key_off + R) : 0)) {
        result[e] = PK_STORE_SKIPPED;
        slot_out[e] = PK_NO_SLOT;
        return;
    }
    if (result[e] != PK_STORE_PENDING) return;
    const unsigned long long w = *reinterpret_cast<const unsigned long long *>(&table[slot_out[e]].slot);
    result[e] = ~(uint32_t)(w >> 32) == (uint32_t)e ? PK_STORE_INSERTED : PK_STORE_PRESENT;
    slot_out[e] = (uint32_t)w;
}

// Table load from device memory in one pass: each 32-byte entry copied whole
// (full-sector writes), a stored entry marked as inserted before any later
// store call (epoch 1, owner 0), and the entry count copied by thread 0.  One
// entry per thread: short blocks, so that kernels of other streams find free
// SM slots while a table is restored beside them.
__global__ void __launch_bounds__(256) k_load_table(pk_entry *table, const pk_entry *src, uint64_t capacity,
                                                    unsigned long long *counter, const unsigned long long *src_count) {
    pk::pdl_wait(table, src, counter, src_count);
    const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i == 0) *counter = __ldcg(src_count);
    if (i < capacity) {
        const uint4 *sp = reinterpret_cast<const uint4 *>(&src[i]);
        const uint4 k = __ldcg(sp);
        uint4 m = __ldcg(sp + 1);  // slot, owner, epoch (low, high)
        if (!is_zero(k)) {
            m.y = 0u;
            m.z = 1u;
            m.w = 0u;
        }
        uint4 *tp = reinterpret_cast<uint4 *>(&table[i]);
        tp[0] = k;
        tp[1] = m;
    }
    pk::pdl_launch_dependents();
}

// After a table load from host memory: every stored entry counts as inserted
// before any later store call (epoch 1; calls on this context use epochs >= 2
// from then on).
__global__ void k_mark_loaded(pk_entry *table, uint64_t capacity) {
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < capacity;
         i += (uint64_t)gridDim.x * blockDim.x) {
        const uint4 k = *reinterpret_cast<const uint4 *>(table[i].k);
        table[i].epoch = is_zero(k) ? 0ull : 1ull;
        table[i].owner = 0u;
    }
}

// ---------------------------------------------------------------------------
// Allocation-free store (pk_store_noalloc).  Same insert-if-absent as the
// store above, for callers that own no libpk context: everything a context
// would hold on the device (entry count, call number) and the per-entry claim
// positions live in this one file-scope array, shared by every call.
// ---------------------------------------------------------------------------
struct NoallocScratch {
    // [0] entries in the table (set by the scan), [1] largest call number
    // found in the table, [2] entries deferred in this call, [3] keys its
    // claims claimed, [4] keys its admission pass claimed, [5] CTAs of the
    // claim kernel done: [0] and [2..5] are the words a context's counter
    // holds at the same indices
    unsigned long long word[6];
    uint32_t pos[PK_NOALLOC_MAX_ENTRIES];  // table position of each PENDING entry
};
static __device__ __align__(256) NoallocScratch g_noalloc_scratch;

// Count the occupied entries and find the latest call number in the table.
__global__ void __launch_bounds__(256)
k_noalloc_scan(const pk_entry *table, uint64_t capacity, NoallocScratch *sc) {
    __shared__ unsigned long long blk_count, blk_epoch;
    if (threadIdx.x == 0) blk_count = blk_epoch = 0;
    __syncthreads();
    unsigned long long cnt = 0, ep = 0;
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < capacity;
         i += (uint64_t)gridDim.x * blockDim.x) {
        const uint4 k = __ldcg(reinterpret_cast<const uint4 *>(table[i].k));
        if (!is_zero(k)) {
            ++cnt;
            const unsigned long long e = __ldcg(&table[i].epoch);
            ep = e > ep ? e : ep;
        }
    }
    atomicAdd_block(&blk_count, cnt);
    atomicMax_block(&blk_epoch, ep);
    __syncthreads();
    if (threadIdx.x == 0) {
        if (blk_count) atomicAdd(&sc->word[0], blk_count);
        atomicMax(&sc->word[1], blk_epoch);
    }
}

// One warp per 32 consecutive entries (list or range mode), as
// k_store_claim; the call number is one past the table's latest and PENDING
// positions go to scratch.
__global__ void __launch_bounds__(256, 4)
k_noalloc_claim(pk_entry *table, uint64_t mask, uint32_t max_probe, uint64_t capacity, NoallocScratch *sc,
                const uint8_t *keys, const uint32_t *slots, uint64_t n,
                const int64_t *key_off, const int32_t *hit, uint32_t R,
                int32_t *result, uint32_t *slot_out, int32_t *status) {
    __shared__ unsigned long long block_sums[2];
    if (threadIdx.x < 2) block_sums[threadIdx.x] = 0;
    __syncthreads();
    const unsigned long long epoch = ld_volatile_u64(&sc->word[1]) + 1ull;
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    bool active = e < n;
    if (key_off) active = in_store_range(key_off, hit, R, n, e) && active;
    const ClaimCtx c{table, mask, max_probe, epoch, claim_mode(sc->word, n, capacity), nullptr};
    int32_t res = PK_STORE_SKIPPED;
    uint32_t out = PK_NO_SLOT;
    ProbeKey s;
    s.pending = false;
    if (active) {
        const uint4 key = __ldcg(reinterpret_cast<const uint4 *>(keys + 32 * e));
        const uint32_t sl = slots[e];
        if (claimable(key, sl, res)) probe_start(s, key, e, mask, sl);
    }
    uint32_t claims = 0, lslot;
    warp_claim<false>(c, s, res, out, lslot, claims);
    if (e < n) {
        result[e] = res;
        if (res == PK_STORE_PENDING) {
            sc->pos[e] = out;
            slot_out[e] = PK_NO_SLOT;
        } else {
            slot_out[e] = out;
        }
        if (res < 0) set_status(status, res);
    }
    count_claims(block_sums, claims, e < n && res == PK_STORE_DEFERRED, sc->word);
    admit_if_last(table, mask, max_probe, capacity, sc->word, epoch, nullptr, keys, slots, n, key_off, R, result,
                  slot_out, sc->pos, status);
}

__global__ void __launch_bounds__(256)
k_noalloc_finalize(const pk_entry *table, const NoallocScratch *sc, uint64_t n, int32_t *result,
                   uint32_t *slot_out) {
    const uint64_t e = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= n || result[e] != PK_STORE_PENDING) return;
    const unsigned long long w = *reinterpret_cast<const unsigned long long *>(&table[sc->pos[e]].slot);
    result[e] = ~(uint32_t)(w >> 32) == (uint32_t)e ? PK_STORE_INSERTED : PK_STORE_PRESENT;
    slot_out[e] = (uint32_t)w;
}

unsigned grid_for(uint64_t n, unsigned block) { return (unsigned)((n + block - 1) / block); }

// Per-request kernels when the batch has many short requests; per-key kernels
// when a few requests carry many keys each (a warp per request would then
// walk them serially).
bool per_request(uint32_t R, uint64_t key_capacity) { return R >= 1024 || key_capacity <= 64ull * R; }

// Resident CTAs of k_lookup_store_req (SMs x CTAs per SM) on the current
// device, computed once per device.
cudaError_t lookup_store_resident(uint64_t *out) {
    static std::mutex mu;
    static uint64_t cache[256] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 256) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!cache[dev]) {
        int sms = 0, per_sm = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_lookup_store_req<true>, kLsBlock, 0);
        if (e != cudaSuccess) return e;
        cache[dev] = (uint64_t)sms * (uint64_t)(per_sm < 1 ? 1 : per_sm);
    }
    *out = cache[dev];
    return cudaSuccess;
}

}  // namespace

cudaError_t pk_launch_load_table(const pk_ctx *ctx, const void *src, cudaStream_t s) {
    const uint64_t blocks = (ctx->capacity + 255) / 256;  // <= 2^23
    const pk_entry *sp = static_cast<const pk_entry *>(src);
    const unsigned long long *cp =
        reinterpret_cast<const unsigned long long *>(static_cast<const uint8_t *>(src) + PK_ENTRY_BYTES * ctx->capacity);
    const cudaError_t e = pk_launch(k_load_table, (unsigned)blocks, 256, s, ctx->table, sp, ctx->capacity,
                                    ctx->counter_dev, cp);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t pk_launch_mark_loaded(const pk_ctx *ctx, cudaStream_t s) {
    const uint64_t blocks = (ctx->capacity + 255) / 256;
    const uint64_t cap = ctx->sm_count ? 16ull * ctx->sm_count : blocks;  // grid-strided: any grid is correct
    k_mark_loaded<<<(unsigned)(blocks < cap ? blocks : cap), 256, 0, s>>>(ctx->table, ctx->capacity);
    return cudaGetLastError();
}

cudaError_t pk_launch_lookup(const pk_ctx *ctx, const uint8_t *keys, const int64_t *key_off, uint32_t R,
                             uint64_t key_capacity, int32_t *hit_chunks, uint32_t *slots, int32_t *status,
                             cudaStream_t s) {
    if (R == 0) return cudaSuccess;
    const uint64_t mask = ctx->capacity - 1;
    cudaError_t e;
    if (per_request(R, key_capacity)) {
        e = pk_launch(k_lookup_req, grid_for(32ull * R, 256), 256, s, (const pk_entry *)ctx->table, mask,
                      ctx->max_probe, keys, key_off, R, key_capacity, slots, hit_chunks, status);
    } else {
        e = key_capacity == 0 ? cudaSuccess
                              : pk_launch(k_lookup, grid_for(key_capacity, 256), 256, s, (const pk_entry *)ctx->table,
                                          mask, ctx->max_probe, keys, key_off, R, key_capacity, slots, status);
        if (e == cudaSuccess)
            e = pk_launch(k_first_miss, grid_for(32ull * R, 256), 256, s, key_off, R, key_capacity,
                          (const uint32_t *)slots, hit_chunks);
    }
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t pk_launch_store(const pk_ctx *ctx, unsigned long long epoch, const uint8_t *keys,
                            const uint32_t *slots, uint64_t n, const int64_t *key_off,
                            const int32_t *hit_chunks, uint32_t R, int32_t *result, uint32_t *slot_out,
                            int32_t *status, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const uint64_t mask = ctx->capacity - 1;
    cudaError_t e;
    if (key_off && R > 0 && per_request(R, n)) {
        e = pk_launch(k_store_claim_req, grid_for(32ull * R, 256), 256, s, ctx->table, mask, ctx->max_probe,
                      ctx->capacity, ctx->counter_dev, epoch, ctx->stamps, keys, slots, n, key_off, hit_chunks, R, result,
                      slot_out, status);
    } else {
        e = pk_launch(k_store_claim, grid_for(n, 256), 256, s, ctx->table, mask, ctx->max_probe, ctx->capacity,
                      ctx->counter_dev, epoch, ctx->stamps, keys, slots, n, key_off, hit_chunks, R, result, slot_out, status);
    }
    if (e == cudaSuccess)
        e = pk_launch(k_store_finalize, grid_for(n, 256), 256, s, (const pk_entry *)ctx->table, n, key_off, R, result,
                      slot_out, ctx->counter_dev);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t pk_launch_lookup_store(const pk_ctx *ctx, unsigned long long epoch, const uint8_t *keys,
                                   const uint32_t *new_slots, const int64_t *key_off, uint32_t R,
                                   uint64_t key_capacity, int32_t *hit_chunks, uint32_t *slots, int32_t *result,
                                   uint32_t *slot_out, int32_t *status, cudaStream_t s) {
    if (R == 0) return cudaSuccess;
    const uint64_t mask = ctx->capacity - 1;
    cudaError_t e;
    if (per_request(R, key_capacity)) {
        uint64_t resident = 0;
        e = lookup_store_resident(&resident);
        if (e != cudaSuccess) return e;
        unsigned long long *tickets = ctx->counter_dev + 1;
        if (R > (kLsBlock / 32) * resident) {  // more requests than resident warps: warps take requests as they finish
            e = cudaMemsetAsync(tickets, 0, sizeof *tickets, s);
            if (e == cudaSuccess)
                e = pk_launch(k_lookup_store_req<true>, (unsigned)resident, kLsBlock, s, ctx->table, mask, ctx->max_probe,
                              ctx->capacity, ctx->counter_dev, epoch, ctx->stamps, keys, new_slots, key_off, R,
                              key_capacity, slots, hit_chunks, result, slot_out, status, tickets);
        } else {
            e = pk_launch(k_lookup_store_req<false>, grid_for(32ull * R, kLsBlock), kLsBlock, s, ctx->table, mask,
                          ctx->max_probe, ctx->capacity, ctx->counter_dev, epoch, ctx->stamps, keys, new_slots, key_off,
                          R, key_capacity, slots, hit_chunks, result, slot_out, status, tickets);
        }
    } else {
        e = key_capacity == 0
                ? cudaSuccess
                : pk_launch(k_lookup_store, grid_for(key_capacity, 256), 256, s, ctx->table, mask, ctx->max_probe,
                            ctx->capacity, ctx->counter_dev, epoch, ctx->stamps, keys, new_slots, key_off, R, key_capacity, slots,
                            result, slot_out, status);
        if (e == cudaSuccess)
            e = pk_launch(k_lookup_store_tail, grid_for(32ull * R, 256), 256, s, key_off, R, key_capacity,
                          (const uint32_t *)slots, hit_chunks, result, slot_out, status);
    }
    if (e == cudaSuccess && key_capacity)
        e = pk_launch(k_store_finalize, grid_for(key_capacity, 256), 256, s, (const pk_entry *)ctx->table,
                      key_capacity, key_off, R, result, slot_out, ctx->counter_dev);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// Device address of the allocation-free store's scratch array, resolved once
// per device (host code cannot use the symbol's host-side name as an address).
static void *noalloc_scratch_addr(int device) {
    static std::mutex mu;
    static void *addr[256] = {};
    if (device < 0 || device >= 256) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[device]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
        addr[device] = p;
    }
    return addr[device];
}

// SMs of a device (0 if the query fails), queried once per device.
static uint32_t device_sms(int device) {
    static std::mutex mu;
    static uint32_t sms[256] = {};
    static bool known[256] = {};
    if (device < 0 || device >= 256) return 0;
    std::lock_guard<std::mutex> lock(mu);
    if (!known[device]) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, device) == cudaSuccess && n > 0)
            sms[device] = (uint32_t)n;
        known[device] = true;
    }
    return sms[device];
}

cudaError_t pk_launch_store_noalloc(pk_entry *table, uint32_t capacity_log2, uint32_t max_probe,
                                    const uint8_t *keys, const uint32_t *slots, uint64_t n, const int64_t *key_off,
                                    const int32_t *hit_chunks, uint32_t R, int32_t *result, uint32_t *slot_out,
                                    int32_t *status, cudaStream_t s) {
    int device = -1;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return e;
    NoallocScratch *sc = static_cast<NoallocScratch *>(noalloc_scratch_addr(device));
    if (!sc) return cudaErrorInvalidSymbol;
    if (n == 0) return cudaSuccess;
    const uint64_t capacity = 1ull << capacity_log2;
    // the counter words must start at zero; pos needs no clearing
    e = cudaMemsetAsync(sc, 0, sizeof sc->word, s);
    if (e != cudaSuccess) return e;
    const uint64_t scan_blocks = (capacity + 255) / 256;
    const uint32_t sms = device_sms(device);
    const uint64_t scan_cap = sms ? 8ull * sms : scan_blocks;  // grid-strided: any grid is correct
    const uint32_t Rm = key_off ? R : 0;
    k_noalloc_scan<<<(unsigned)(scan_blocks < scan_cap ? scan_blocks : scan_cap), 256, 0, s>>>(table, capacity, sc);
    k_noalloc_claim<<<grid_for(n, 256), 256, 0, s>>>(table, capacity - 1, max_probe, capacity, sc, keys, slots, n,
                                                      key_off, hit_chunks, Rm, result, slot_out, status);
    k_noalloc_finalize<<<grid_for(n, 256), 256, 0, s>>>(table, sc, n, result, slot_out);
    return cudaGetLastError();
}
