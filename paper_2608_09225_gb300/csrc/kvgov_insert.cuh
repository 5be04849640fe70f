// kvgov_insert.cuh -- the per-key insert protocol of the prefix-cache table
// (slot encoding and protocol as described in kvgov_table.cu and
// include/kvgov.h), shared by the insert kernels and the arrival-order
// insert.
#pragma once
#include <cstdint>

#include "kvgov_lookup.cuh"
#include "kvgov_stash.cuh"

namespace kvgov_dev {

__device__ __forceinline__ unsigned long long ld_relaxed(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];\n" : "=l"(v) : "l"(p) : "memory");
    return v;
}
// A plain (weak) 16-byte load, which the SM's L1 may serve.  Within a kernel
// L1 is not kept coherent with other SMs' writes, so such a load can return
// an older value.  The protocol applies it only to words that are written
// once from zero, where an older value is zero and sends the thread to the
// coherent path; on hot keys it keeps the repeated reads in L1.
__device__ __forceinline__ ulonglong2 ld_plain2(const unsigned long long *p) {
    ulonglong2 v;
    asm volatile("ld.global.v2.u64 {%0, %1}, [%2];\n" : "=l"(v.x), "=l"(v.y) : "l"(p) : "memory");
    return v;
}
// Both words of a 16-byte-aligned pair in one store.  Each word is written
// once, from zero, so a reader that sees one word and not the other still
// sees a zero word and waits.
__device__ __forceinline__ void st_relaxed2(unsigned long long *p, unsigned long long a, unsigned long long b) {
    asm volatile("st.relaxed.gpu.global.v2.u64 [%0], {%1, %2};\n" ::"l"(p), "l"(a), "l"(b) : "memory");
}

// 128-bit compare-and-swap of the 16-byte-aligned pair p[0..1]: if it holds
// (c0, c1) it becomes (n0, n1); the previous value is returned in (o0, o1).
__device__ __forceinline__ void cas128(unsigned long long *p, unsigned long long c0, unsigned long long c1,
                                       unsigned long long n0, unsigned long long n1, unsigned long long &o0,
                                       unsigned long long &o1) {
    asm volatile("{\n\t.reg .b128 c, n, o;\n\t"
                 "mov.b128 c, {%2, %3};\n\t"
                 "mov.b128 n, {%4, %5};\n\t"
                 "atom.relaxed.gpu.global.cas.b128 o, [%6], c, n;\n\t"
                 "mov.b128 {%0, %1}, o;\n\t}"
                 : "=l"(o0), "=l"(o1)
                 : "l"(c0), "l"(c1), "l"(n0), "l"(n1), "l"(p)
                 : "memory");
}

enum InsertResult { kNew = 0, kDuplicate = 1, kFull = 2, kTimeout = 3 };

// Arrival-order serving (kvgov_arrival.cu): the slot_of entry of a block
// whose key is not in the table, and the mark the insert sets on a block
// whose owner it has already settled (the owner min clears it).
constexpr uint32_t kNoSlot = 0xffffffffu;
constexpr uint32_t kSettled = 0x80000000u;

// Insert the non-zero key k (w0..w3) with the protocol described in
// kvgov_table.cu; keys the main slots cannot hold go to the side store
// (kvgov_stash.cuh).  On kNew and kDuplicate, *pos receives the key's handle:
// the slot that holds it, or capacity + 8 + its side-store entry.
// start: the walk begins start slots past the home slot -- the caller has
// seen each slot before it holding a complete first half (both words non-
// zero) other than the key's, which is final.
__device__ __forceinline__ InsertResult insert_one(unsigned long long *slots, unsigned long long mask,
                                                   const unsigned long long k[4], uint32_t spin_limit,
                                                   unsigned long long *pos_out = nullptr,
                                                   unsigned long long start = 0) {
    if (key_in_stash(k[0], k[1], k[2], k[3])) {
        const StashResult r = stash_insert(slots, mask, k[0], k[1], k[2], k[3], spin_limit);
        if (pos_out && (r.res == kNew || r.res == kDuplicate)) *pos_out = r.pos;
        return static_cast<InsertResult>(r.res);
    }
    const unsigned long long window = probe_window(mask);
    unsigned long long pos = (k[0] + start) & mask;
    for (unsigned long long n = start; n < window; ++n, pos = (pos + 1) & mask) {
        unsigned long long *slot = slots + 4 * pos;
        unsigned long long o0 = 0ull, o1 = 0ull;
        // Look first (measured: it turns the step after a cache flush, where
        // every request inserts the same shared-prefix blocks, from ~377 to
        // ~70 us for +5 us on an ordinary step).  A slot's first half is written once, from (0, 0) to
        // its final value, so a read racing that write (or an older copy in
        // L1) can only show a zero word; a read with both words non-zero is
        // the final value and needs no atomic (another key: walk on; our
        // first half: compare).
        const ulonglong2 seen = ld_plain2(slot);
        o0 = seen.x;
        o1 = seen.y;
        if (o0 == 0ull || o1 == 0ull) {
            cas128(slot, 0ull, 0ull, k[0], k[1], o0, o1);
            if ((o0 | o1) == 0ull) {                 // claimed: write the second half
                st_relaxed2(slot + 2, k[2], k[3]);
                if (pos_out) *pos_out = pos;
                return kNew;
            }
        }
        if (o0 != k[0] || o1 != k[1]) continue;      // another key
        // The second half is written once from zero too: a plain read with
        // both words non-zero is final; otherwise wait on coherent reads.
        const ulonglong2 second = ld_plain2(slot + 2);
        unsigned long long w2 = second.x, w3 = second.y;
        for (uint32_t spins = 0; w2 == 0ull || w3 == 0ull; ++spins) {
            if (spins >= spin_limit) return kTimeout;
            __nanosleep(100);
            w2 = ld_relaxed(slot + 2);
            w3 = ld_relaxed(slot + 3);
        }
        if (w2 == k[2] && w3 == k[3]) {
            if (pos_out) *pos_out = pos;
            return kDuplicate;
        }
    }
    return kFull;
}

// Insert counts: warp reduction, shared-memory accumulation, and the CTA's
// last warp to finish publishes them (no barrier: early warps just exit).
__device__ __forceinline__ void publish_counts(unsigned my_new, unsigned my_flags, unsigned *s_new, unsigned *s_flags,
                                               unsigned *s_done, unsigned long long *n_new, uint32_t *status) {
    const unsigned w_new = __reduce_add_sync(0xffffffffu, my_new);
    const unsigned w_flags = __reduce_or_sync(0xffffffffu, my_flags);
    if ((threadIdx.x & 31) == 0) {
        if (w_new) atomicAdd(s_new, w_new);
        if (w_flags) atomicOr(s_flags, w_flags);
        __threadfence_block();
        if (atomicAdd(s_done, 1u) == blockDim.x / 32 - 1) {
            const unsigned t_new = atomicAdd(s_new, 0u), t_flags = atomicOr(s_flags, 0u);
            if (t_new && n_new) atomicAdd(n_new, (unsigned long long)t_new);
            if (t_flags && status) atomicOr(status, t_flags);
        }
    }
}

__device__ __forceinline__ void count_insert(InsertResult res, unsigned &my_new, unsigned &my_flags) {
    switch (res) {
    case kNew: ++my_new; break;
    case kDuplicate: break;
    case kFull: my_flags |= KVGOV_F_TABLE_FULL; break;
    default: my_flags |= KVGOV_F_TIMEOUT; break;
    }
}

}  // namespace kvgov_dev
