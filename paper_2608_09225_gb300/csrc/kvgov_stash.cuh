// kvgov_stash.cuh -- the table's side store: the keys that the main slots'
// claim protocol cannot hold (layout in include/kvgov.h, KVGOV_STASH_*).
//
// A main slot is claimed by a 128-bit compare-and-swap of the key's first 16
// bytes from zero, and its second half is then written with plain stores; a
// reader that sees a zero 8-byte word in the second half waits for the
// writer.  So a key whose first half is zero (it would look empty) or whose
// second half holds a zero 8-byte word (it would look half-written) cannot
// live in a main slot.  Such keys -- any other 32-byte key but the all-zero
// one, which the library refuses -- go to this side store after the
// `capacity` main slots, so that the table holds every non-zero key.  A
// SHA-256 digest lands here with probability about 2^-63, so the store is
// small and its protocol is simple rather than fast:
//
//   slot 0 (bytes 0-3)  count: entry indices handed out so far (saturates at
//                       KVGOV_STASH_KEYS; zeroed by kvgov_table_init)
//   bytes 32-255        state of entry e (u32 at byte 32 + 4e): 0 = being
//                       written, kStashLive = holds its key
//   slots 8 .. 63       entry e's key in slot 8 + e; its handle (the slot
//                       index the arrival-order owner array uses) is
//                       capacity + 8 + e
//
// Insert: look through the entries handed out so far, waiting for each to
// be published; if the key is live in one, it is a duplicate.  Otherwise
// take the next entry with a compare-and-swap of the count from the value
// the scan covered to one more: it succeeds only if no entry was handed out
// since, so the thread has seen every entry below its own; if another
// thread took one meanwhile, scan the new entries and try again.  The
// winner writes the key and publishes the entry live with a release store,
// with no wait in between, so a thread that waits for an entry waits a few
// instructions of another thread's (each wait is bounded all the same:
// spin_limit re-reads, then KVGOV_F_TIMEOUT).  Every entry handed out holds
// a distinct key, and two inserts of one key leave it in one entry, in any
// interleaving.  Lookups run while the table does not change and scan the
// live entries.
#pragma once
#include <cstdint>

#include "../../include/kvgov.h"

namespace kvgov_dev {

constexpr int kStashHeaderSlots = 8;
constexpr uint32_t kStashLive = 1u;
static_assert(kStashHeaderSlots + KVGOV_STASH_KEYS == KVGOV_STASH_SLOTS, "side store layout");
static_assert(32 + 4 * KVGOV_STASH_KEYS <= 32 * kStashHeaderSlots, "entry states fit the header");

// Keys the main slots cannot hold (the all-zero key excluded by the caller).
__device__ __forceinline__ bool key_in_stash(unsigned long long k0, unsigned long long k1, unsigned long long k2,
                                             unsigned long long k3) {
    return (k0 | k1) == 0ull || k2 == 0ull || k3 == 0ull;
}

__device__ __forceinline__ bool key_is_zero(const unsigned long long k[4]) {
    return (k[0] | k[1] | k[2] | k[3]) == 0ull;
}

__device__ __forceinline__ uint32_t stash_ld_acquire(const uint32_t *p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];\n" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void stash_st_release(uint32_t *p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;\n" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned long long stash_ld_relaxed(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];\n" : "=l"(v) : "l"(p) : "memory");
    return v;
}

struct StashResult {
    int res;                   // InsertResult of kvgov_insert.cuh: 0 new, 1 duplicate, 2 full, 3 timeout
    unsigned long long pos;    // the key's handle (new or duplicate)
};

// Insert into the side store of the table whose main slots are
// slots[0 .. mask]; the key is non-zero and key_in_stash.  Kept out of line:
// the hot kernels reach it only for those keys.
static __device__ __noinline__ StashResult stash_insert(unsigned long long *slots, unsigned long long mask,
                                                        unsigned long long k0, unsigned long long k1,
                                                        unsigned long long k2, unsigned long long k3,
                                                        uint32_t spin_limit) {
    unsigned long long *base = slots + 4 * (mask + 1);
    uint32_t *count = reinterpret_cast<uint32_t *>(base);
    uint32_t *state = count + 8;
    unsigned long long *keys = base + 4 * kStashHeaderSlots;
    const unsigned long long first = mask + 1 + kStashHeaderSlots;    // handle of entry 0
    // Wait (bounded) until entry e is published; false on timeout.
    auto published = [&](int e) -> bool {
        for (uint32_t spins = 0;; ++spins) {
            if (stash_ld_acquire(state + e) == kStashLive) return true;
            if (spins >= spin_limit) return false;
            __nanosleep(100);
        }
    };
    auto holds = [&](int e) {
        const unsigned long long *w = keys + 4 * e;
        return stash_ld_relaxed(w) == k0 && stash_ld_relaxed(w + 1) == k1 && stash_ld_relaxed(w + 2) == k2 &&
               stash_ld_relaxed(w + 3) == k3;
    };
    uint32_t seen = 0;                                       // entries [0, seen) hold other keys
    // at most KVGOV_STASH_KEYS entries are ever handed out, and each failed
    // compare-and-swap below means one was: the loop ends
    for (;;) {
        uint32_t cur = stash_ld_acquire(count);
        if (cur > (uint32_t)KVGOV_STASH_KEYS) cur = KVGOV_STASH_KEYS;
        for (; seen < cur; ++seen) {
            if (!published((int)seen)) return {3, 0ull};
            if (holds((int)seen)) return {1, first + seen};
        }
        if (cur >= (uint32_t)KVGOV_STASH_KEYS) return {2, 0ull};
        if (atomicCAS(count, cur, cur + 1u) != cur) continue;   // another entry was handed out: scan it
        unsigned long long *w = keys + 4 * cur;
        w[0] = k0;
        w[1] = k1;
        w[2] = k2;
        w[3] = k3;
        stash_st_release(state + cur, kStashLive);          // the key's words are visible before the state
        return {0, first + cur};
    }
}

// Is the key (q0, q1: bytes 0-15, 16-31) live in the side store?  For
// lookups while the table does not change.
static __device__ __noinline__ bool stash_lookup(const uint4 *slots, unsigned long long mask, uint4 q0, uint4 q1) {
    const uint4 *base = slots + 2 * (mask + 1);
    const uint32_t *count = reinterpret_cast<const uint32_t *>(base);
    const uint32_t *state = count + 8;
    const uint32_t seen = __ldg(count);
    const int n = seen < (uint32_t)KVGOV_STASH_KEYS ? (int)seen : KVGOV_STASH_KEYS;
    for (int e = 0; e < n; ++e) {
        if (__ldg(state + e) != kStashLive) continue;
        const uint4 a = __ldg(base + 2 * (kStashHeaderSlots + e)), b = __ldg(base + 2 * (kStashHeaderSlots + e) + 1);
        if (a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w && b.x == q1.x && b.y == q1.y && b.z == q1.z &&
            b.w == q1.w)
            return true;
    }
    return false;
}

// stash_lookup returning the key's handle (capacity + 8 + its entry), or -1.
static __device__ __noinline__ long long stash_lookup_handle(const uint4 *slots, unsigned long long mask, uint4 q0,
                                                             uint4 q1) {
    const uint4 *base = slots + 2 * (mask + 1);
    const uint32_t *count = reinterpret_cast<const uint32_t *>(base);
    const uint32_t *state = count + 8;
    const uint32_t seen = __ldg(count);
    const int n = seen < (uint32_t)KVGOV_STASH_KEYS ? (int)seen : KVGOV_STASH_KEYS;
    for (int e = 0; e < n; ++e) {
        if (__ldg(state + e) != kStashLive) continue;
        const uint4 a = __ldg(base + 2 * (kStashHeaderSlots + e)), b = __ldg(base + 2 * (kStashHeaderSlots + e) + 1);
        if (a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w && b.x == q1.x && b.y == q1.y && b.z == q1.z &&
            b.w == q1.w)
            return (long long)(mask + 1 + kStashHeaderSlots + e);
    }
    return -1;
}

}  // namespace kvgov_dev
