// kvgov_lookup.cuh -- read-only lookup of a 32-byte key in the prefix-cache
// table (slot encoding and probe window as described in kvgov_table.cu and
// include/kvgov.h), shared by the probe kernels and the fused chain + probe
// kernel.  Exact while the table does not change.  While inserts run (the
// chain launch that carries the previous batch's insert), a slot only goes
// from empty to claimed to complete and never changes its key, so a lookup
// can miss a key that is being inserted but never finds an absent one.
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

// lookup() returning the key's handle -- the slot that holds it, or
// capacity + 8 + its side-store entry -- or -1 if it is absent.
__device__ __forceinline__ long long lookup_handle(const uint4 *__restrict__ slots, unsigned long long mask, uint4 q0,
                                                   uint4 q1) {
    const unsigned long long k0 = u64_of(q0.x, q0.y), k1 = u64_of(q0.z, q0.w);
    if (key_in_stash(k0, k1, u64_of(q1.x, q1.y), u64_of(q1.z, q1.w)))
        return stash_lookup_handle(slots, mask, q0, q1);
    const unsigned long long window = probe_window(mask);
    unsigned long long pos = k0 & mask;
    for (unsigned long long n = 0; n < window; ++n, pos = (pos + 1) & mask) {
        const uint4 a = __ldg(slots + 2 * pos);
        if ((a.x | a.y | a.z | a.w) == 0u) return -1;
        if (a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w) {
            const uint4 b = __ldg(slots + 2 * pos + 1);
            if (b.x == q1.x && b.y == q1.y && b.z == q1.z && b.w == q1.w) return (long long)pos;
        }
    }
    return -1;
}

// The lookup of kvgov_chain_hash_serve: 1 = the key is in the table with a
// generation in [floor, g) (cached for this batch), 0 = it is in the table
// with another generation (added by this batch: nothing to insert), -1 = not
// found.  On -1, *start is where an insert of the key may begin its walk:
// the offset from the home slot of the first slot not seen holding a
// complete first half (both words non-zero) other than the key's.  The home
// slot's generation is read with the home slot, where most keys are found.
__device__ __forceinline__ int lookup_serve(const uint4 *__restrict__ slots, unsigned long long mask,
                                            const uint32_t *gen, uint32_t floor, uint32_t g, uint4 q0, uint4 q1,
                                            unsigned long long *start) {
    *start = 0;
    const unsigned long long k0 = u64_of(q0.x, q0.y), k1 = u64_of(q0.z, q0.w);
    if (key_in_stash(k0, k1, u64_of(q1.x, q1.y), u64_of(q1.z, q1.w))) {
        const long long h = stash_lookup_handle(slots, mask, q0, q1);
        if (h < 0) return -1;
        const uint32_t gv = gen[h];
        return gv >= floor && gv < g ? 1 : 0;
    }
    const unsigned long long window = probe_window(mask);
    const unsigned long long home = k0 & mask;
    const uint32_t gv_home = gen[home];
    bool open = true;                                   // every slot so far: a complete first half, not the key's
    unsigned long long pos = home;
    for (unsigned long long n = 0; n < window; ++n, pos = (pos + 1) & mask) {
        const uint4 a = __ldg(slots + 2 * pos);
        if ((a.x | a.y | a.z | a.w) == 0u) {
            if (open) *start = n;
            return -1;
        }
        const bool mine = a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w;
        if (mine) {
            const uint4 b = __ldg(slots + 2 * pos + 1);
            if (b.x == q1.x && b.y == q1.y && b.z == q1.z && b.w == q1.w) {
                const uint32_t gv = n == 0 ? gv_home : gen[pos];
                return gv >= floor && gv < g ? 1 : 0;
            }
        }
        if (open && (mine || (a.x | a.y) == 0u || (a.z | a.w) == 0u)) {
            *start = n;                                 // an insert must look at this slot itself
            open = false;
        }
    }
    if (open) *start = window;
    return -1;
}

// The home slot of the key q0 || q1.
__device__ __forceinline__ unsigned long long home_slot(uint4 q0, unsigned long long mask) {
    return u64_of(q0.x, q0.y) & mask;
}

// The first S slots of a walk (S = 1: the home slot a, b; S = 2: also the
// next slot c, d), read by the caller: 1 = the key is there, 0 = the walk
// ended without it, -1 = all S slots hold other keys and the walk goes on at
// home + S (warp_finish_walks).  The window is at least 32 slots (capacity
// is a power of two >= 32), so it never ends inside the first two.
template <int S>
__device__ __forceinline__ int walk_start(const uint4 *__restrict__ slots, unsigned long long mask, uint4 q0,
                                          uint4 q1, uint4 a, uint4 b, uint4 c, uint4 d) {
    if (key_in_stash(u64_of(q0.x, q0.y), u64_of(q0.z, q0.w), u64_of(q1.x, q1.y), u64_of(q1.z, q1.w)))
        return stash_lookup(slots, mask, q0, q1) ? 1 : 0;    // not in the main slots
    if ((a.x | a.y | a.z | a.w) == 0u) return 0;
    if (a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w && b.x == q1.x && b.y == q1.y && b.z == q1.z &&
        b.w == q1.w)
        return 1;
    if (S == 1) return -1;
    if ((c.x | c.y | c.z | c.w) == 0u) return 0;
    if (c.x == q0.x && c.y == q0.y && c.z == q0.z && c.w == q0.w && d.x == q1.x && d.y == q1.y && d.z == q1.z &&
        d.w == q1.w)
        return 1;
    return -1;
}

// A walk_start<S> state of -1, finished by this lane alone: two slots a
// memory round trip from home + S to the key, an empty slot or the end of
// the window.  1 = the key is there, 0 = it is not.
template <int S>
__device__ __forceinline__ int walk_on(const uint4 *__restrict__ slots, unsigned long long mask, uint4 q0, uint4 q1) {
    const unsigned long long window = probe_window(mask);   // even: capacity is a power of two >= 32
    for (unsigned long long n = S, pos = (home_slot(q0, mask) + S) & mask; n < window; n += 2) {
        const unsigned long long nxt = (pos + 1) & mask;
        const uint4 a = __ldg(slots + 2 * pos), b = __ldg(slots + 2 * pos + 1);
        const uint4 c = __ldg(slots + 2 * nxt), d = __ldg(slots + 2 * nxt + 1);
        if ((a.x | a.y | a.z | a.w) == 0u) return 0;
        if (a.x == q0.x && a.y == q0.y && a.z == q0.z && a.w == q0.w && b.x == q1.x && b.y == q1.y &&
            b.z == q1.z && b.w == q1.w)
            return 1;
        if (n + 1 == window) return 0;                       // S = 1: the window's last slot was a
        if ((c.x | c.y | c.z | c.w) == 0u) return 0;
        if (c.x == q0.x && c.y == q0.y && c.z == q0.z && c.w == q0.w && d.x == q1.x && d.y == q1.y &&
            d.z == q1.z && d.w == q1.w)
            return 1;
        pos = (pos + 2) & mask;
    }
    return 0;
}

// Finish together the walks of the lanes whose walk_start<S> state st is -1
// (every lane of the warp calls it; the others pass 0 or 1 and get it back).
// In each memory round trip the k walks still going share the warp's 32
// lanes, 32 / 2^ceil(log2 k) consecutive lanes each, every lane reading one
// slot of its walk's next stretch (both halves); the first slot of the
// stretch that is empty or holds the key ends the walk.  At load factor 0.5
// one walk in ten reads more than four slots and one in a hundred more than
// twelve: walked two slots a trip, each lane on its own, a warp's 32 walks
// would take as many trips as the longest of them, about six; shared out,
// a walk that goes on takes one or two.  Same result as lookup().
template <int S>
__device__ __forceinline__ int warp_finish_walks(const uint4 *__restrict__ slots, unsigned long long mask, uint4 q0,
                                                 uint4 q1, int st) {
    const int lane = threadIdx.x & 31;
    const unsigned window = (unsigned)probe_window(mask);
    unsigned long long pos = (home_slot(q0, mask) + S) & mask;   // the walk's next slot
    unsigned n = S;                                              // slots walked so far
    unsigned go = __ballot_sync(0xffffffffu, st < 0);
    while (go) {                                                 // warp-uniform
        const int k = __popc(go);
        const int lg = k == 1 ? 0 : 32 - __clz(k - 1);
        const int lw = 32 >> lg;                                 // lanes per walk
        const int wi = lane >> (5 - lg), j = lane & (lw - 1);    // this lane's walk, its slot in the stretch
        const int src = wi < k ? __fns(go, 0, wi + 1) : lane;    // the lane whose walk it is
        uint4 s0, s1;
        s0.x = __shfl_sync(0xffffffffu, q0.x, src); s0.y = __shfl_sync(0xffffffffu, q0.y, src);
        s0.z = __shfl_sync(0xffffffffu, q0.z, src); s0.w = __shfl_sync(0xffffffffu, q0.w, src);
        s1.x = __shfl_sync(0xffffffffu, q1.x, src); s1.y = __shfl_sync(0xffffffffu, q1.y, src);
        s1.z = __shfl_sync(0xffffffffu, q1.z, src); s1.w = __shfl_sync(0xffffffffu, q1.w, src);
        const unsigned long long spos = __shfl_sync(0xffffffffu, pos, src);
        const unsigned sn = __shfl_sync(0xffffffffu, n, src);
        bool end = false, found = false;
        if (wi < k && sn + (unsigned)j < window) {
            const unsigned long long sp = (spos + (unsigned long long)j) & mask;
            const uint4 a = __ldg(slots + 2 * sp), b = __ldg(slots + 2 * sp + 1);
            if ((a.x | a.y | a.z | a.w) == 0u) {
                end = true;
            } else if (a.x == s0.x && a.y == s0.y && a.z == s0.z && a.w == s0.w && b.x == s1.x && b.y == s1.y &&
                       b.z == s1.z && b.w == s1.w) {
                end = found = true;
            }
        }
        const unsigned eb = __ballot_sync(0xffffffffu, end), fb = __ballot_sync(0xffffffffu, found);
        if (st < 0) {
            const int my = __popc(go & ((1u << lane) - 1u));     // this walk's rank among those going
            const unsigned e = (eb >> (my * lw)) & (lw == 32 ? 0xffffffffu : ((1u << lw) - 1u));
            if (e) {
                st = (int)((fb >> (my * lw + __ffs((int)e) - 1)) & 1u);
            } else {
                pos = (pos + (unsigned long long)lw) & mask;
                n += (unsigned)lw;
                if (n >= window) st = 0;                         // the window holds no empty slot and not the key
            }
        }
        go = __ballot_sync(0xffffffffu, st < 0);
    }
    return st;
}

}  // namespace kvgov_dev
