// kvgov_lookup.cuh -- read-only lookup of a 32-byte key in the prefix-cache
// table (slot encoding and probe window as described in kvgov_table.cu and
// include/kvgov.h), shared by the probe kernels and the fused chain + probe
// kernel.  The table must not change while a lookup runs.
#pragma once
#include <cstdint>

#include "../../include/kvgov.h"
#include "kvgov_stash.cuh"

namespace kvgov_dev {

__device__ __forceinline__ unsigned long long u64_of(uint32_t lo, uint32_t hi) {
    return (unsigned long long)lo | ((unsigned long long)hi << 32);
}

// Slots a key may occupy past its home slot: min(capacity, KVGOV_PROBE_WINDOW).
__device__ __forceinline__ unsigned long long probe_window(unsigned long long mask) {
    return mask < KVGOV_PROBE_WINDOW - 1 ? mask + 1 : (unsigned long long)KVGOV_PROBE_WINDOW;
}

// Is the key q0 || q1 (bytes 0-15, 16-31, as stored) in the table?  Slots are
// read through the read-only path, the second half of a slot only when the
// first matches (fewer loads: the fused chain kernel, whose lookups hide
// behind other warps' hashing).
__device__ __forceinline__ bool lookup(const uint4 *__restrict__ slots, unsigned long long mask, uint4 q0, uint4 q1) {
    const unsigned long long k0 = u64_of(q0.x, q0.y), k1 = u64_of(q0.z, q0.w);
    if (key_in_stash(k0, k1, u64_of(q1.x, q1.y), u64_of(q1.z, q1.w)))
        return stash_lookup(slots, mask, q0, q1);    // not in the main slots
    const unsigned long long window = probe_window(mask);
    unsigned long long pos = k0 & mask;
    for (unsigned long long n = 0; n < window; ++n, pos = (pos + 1) & mask) {
        const uint4 a = __ldg(slots + 2 * pos);
        if ((a.x | a.y | a.z | a.w) == 0u) return false;   // empty slot ends the walk
        if (a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w) {
            const uint4 b = __ldg(slots + 2 * pos + 1);
            if (b.x == q1.x && b.y == q1.y && b.z == q1.z && b.w == q1.w) return true;
        }
    }
    return false;
}

// The home slot of the key q0 || q1.
__device__ __forceinline__ unsigned long long home_slot(uint4 q0, unsigned long long mask) {
    return u64_of(q0.x, q0.y) & mask;
}

// lookup() whose first slot, the key's home slot (both halves a, b), the
// caller has read already: the probe kernels issue the home-slot loads of
// several keys together and finish each walk after.  Same result as
// lookup().
__device__ __forceinline__ bool lookup_from_home(const uint4 *__restrict__ slots, unsigned long long mask, uint4 q0,
                                                 uint4 q1, uint4 a, uint4 b) {
    if (key_in_stash(u64_of(q0.x, q0.y), u64_of(q0.z, q0.w), u64_of(q1.x, q1.y), u64_of(q1.z, q1.w)))
        return stash_lookup(slots, mask, q0, q1);    // not in the main slots
    const unsigned long long window = probe_window(mask);
    unsigned long long pos = home_slot(q0, mask);
    for (unsigned long long n = 1;; ++n) {
        if ((a.x | a.y | a.z | a.w) == 0u) return false;   // empty slot ends the walk
        if (a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w && b.x == q1.x && b.y == q1.y &&
            b.z == q1.z && b.w == q1.w)
            return true;
        if (n == window) return false;
        pos = (pos + 1) & mask;
        a = __ldg(slots + 2 * pos);
        b = __ldg(slots + 2 * pos + 1);
    }
}

// lookup() whose first two slots, the key's home slot (a, b) and the next
// one (c, d), the caller has read already (four independent loads, one
// memory round trip); the walk goes on two slots per round trip.  A walk
// of up to two slots -- most hits and, at load factor 0.5, half the misses
// -- then costs one round trip.  Same result as lookup().
__device__ __forceinline__ bool lookup_from_pair(const uint4 *__restrict__ slots, unsigned long long mask, uint4 q0,
                                                 uint4 q1, uint4 a, uint4 b, uint4 c, uint4 d) {
    if (key_in_stash(u64_of(q0.x, q0.y), u64_of(q0.z, q0.w), u64_of(q1.x, q1.y), u64_of(q1.z, q1.w)))
        return stash_lookup(slots, mask, q0, q1);    // not in the main slots
    const unsigned long long window = probe_window(mask);   // even: capacity is a power of two >= 32
    unsigned long long pos = home_slot(q0, mask);
    for (unsigned long long n = 2;; n += 2) {
        if ((a.x | a.y | a.z | a.w) == 0u) return false;   // empty slot ends the walk
        if (a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w && b.x == q1.x && b.y == q1.y &&
            b.z == q1.z && b.w == q1.w)
            return true;
        if ((c.x | c.y | c.z | c.w) == 0u) return false;
        if (c.x == q0.x && c.y == q0.y && c.z == q0.z && c.w == q0.w && d.x == q1.x && d.y == q1.y &&
            d.z == q1.z && d.w == q1.w)
            return true;
        if (n == window) return false;
        pos = (pos + 2) & mask;
        const unsigned long long nxt = (pos + 1) & mask;
        a = __ldg(slots + 2 * pos);
        b = __ldg(slots + 2 * pos + 1);
        c = __ldg(slots + 2 * nxt);
        d = __ldg(slots + 2 * nxt + 1);
    }
}

}  // namespace kvgov_dev
