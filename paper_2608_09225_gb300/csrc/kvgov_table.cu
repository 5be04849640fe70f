// kvgov_table.cu -- the block prefix-cache index: a power-of-two open-
// addressing table of 32-byte digests (kvgov_table_init, kvgov_insert,
// kvgov_probe).
//
// Paper: section 2.1 (a lookup matches the longest common prefix from
// position 0, truncated to a block boundary), Table 1 row 1 (a block prefix
// cache; the probe learns the first k matched blocks), section 4.1 (an
// adversary's probes only populate its own namespace), section 5.7 (a
// divergence at token i invalidates every block from floor(i/B) on).
//
// Slot encoding: four little-endian u64 words w0..w3 = the key verbatim.
// w0 == 0 marks an empty slot and w0 == ~0 a slot claimed by an insert that
// has not yet published the key; keys with those first words are refused.
// Home slot = w0 & (capacity - 1); collisions go to the next slot (linear
// probing, wrapping).
//
// Insert protocol (one key per thread): CAS w0 from 0 to the claim marker,
// store w1..w3, then store w0 = key with release semantics.  A thread that
// meets a claimed slot re-reads it with acquire loads, a bounded number of
// times, until the owner publishes; then it compares the full key (equal =
// duplicate, done; different = keep probing).  Two inserts of one key in one
// batch therefore store it once.
//
// Probe: G lanes of a warp serve one request.  The lanes look up the next G
// consecutive blocks in parallel; a ballot over the window's misses gives the
// first miss (the prefix length) and ends the request, else the window moves
// on.  A request of n_b blocks takes ceil((L+1)/G) rounds of two dependent
// memory accesses (digest, slot); lookups past the first miss inside the last
// window are wasted, which costs bandwidth but not latency.
#include <atomic>

#include "kvgov_internal.cuh"

namespace {

using namespace kvgov_dev;

constexpr unsigned long long kClaimed = ~0ull;
constexpr uint32_t kDefaultSpin = 1u << 23;
std::atomic<uint32_t> g_spin_limit{kDefaultSpin};

__device__ __forceinline__ unsigned long long ld_acquire(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];\n" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ unsigned long long ld_relaxed(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];\n" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ ulonglong2 ld_relaxed2(const unsigned long long *p) {
    ulonglong2 v;
    asm volatile("ld.relaxed.gpu.global.v2.u64 {%0, %1}, [%2];\n" : "=l"(v.x), "=l"(v.y) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_relaxed(unsigned long long *p, unsigned long long v) {
    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;\n" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ void st_release(unsigned long long *p, unsigned long long v) {
    asm volatile("st.release.gpu.global.u64 [%0], %1;\n" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ unsigned long long u64_of(uint32_t lo, uint32_t hi) {
    return (unsigned long long)lo | ((unsigned long long)hi << 32);
}

// ---------------------------------------------------------------------------
__global__ void table_init_kernel(uint4 *__restrict__ slots, unsigned long long n_vec) {
    for (unsigned long long i = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; i < n_vec;
         i += (unsigned long long)gridDim.x * blockDim.x)
        slots[i] = make_uint4(0u, 0u, 0u, 0u);
}

// ---------------------------------------------------------------------------
constexpr int kInsertThreads = 256;

enum InsertResult { kNew = 0, kDuplicate = 1, kFull = 2, kTimeout = 3 };

__device__ InsertResult insert_one(unsigned long long *slots, unsigned long long mask, const unsigned long long k[4],
                                   uint32_t spin_limit) {
    unsigned long long pos = k[0] & mask;
    for (unsigned long long n = 0; n <= mask; ++n, pos = (pos + 1) & mask) {
        unsigned long long *slot = slots + 4 * pos;
        // One 32-byte look at the slot.  A slot is written once (claim, tail,
        // publish) and never changes afterwards, so a full match on these
        // unordered reads can only be the key itself: a duplicate.
        const ulonglong2 lo = ld_relaxed2(slot), hi = ld_relaxed2(slot + 2);
        unsigned long long w0 = lo.x;
        if (w0 == k[0] && lo.y == k[1] && hi.x == k[2] && hi.y == k[3]) return kDuplicate;
        if (w0 == 0ull) {
            const unsigned long long old = atomicCAS(slot, 0ull, kClaimed);
            if (old == 0ull) {
                st_relaxed(slot + 1, k[1]);
                st_relaxed(slot + 2, k[2]);
                st_relaxed(slot + 3, k[3]);
                st_release(slot, k[0]);
                return kNew;
            }
            w0 = old;
        }
        if (w0 == kClaimed || w0 == k[0]) {
            // claimed but not yet published, or our first word with a tail
            // that may have been read before it was written: wait for the
            // publication (bounded) and compare again with acquire ordering
            uint32_t spins = 0;
            while ((w0 = ld_acquire(slot)) == kClaimed) {
                if (++spins >= spin_limit) return kTimeout;
                __nanosleep(100);
            }
            if (w0 == k[0]) {
                const ulonglong2 t = ld_relaxed2(slot + 2);
                if (ld_relaxed(slot + 1) == k[1] && t.x == k[2] && t.y == k[3]) return kDuplicate;
            }
        }
    }
    return kFull;
}

__global__ void __launch_bounds__(kInsertThreads) insert_kernel(unsigned long long *__restrict__ slots,
                                                                unsigned long long mask,
                                                                const uint4 *__restrict__ keys, long long n_keys,
                                                                unsigned long long *n_new, uint32_t *status,
                                                                uint32_t spin_limit) {
    __shared__ unsigned int s_new, s_flags, s_done;
    if (threadIdx.x == 0) { s_new = 0; s_flags = 0; s_done = 0; }
    __syncthreads();
    const long long stride = (long long)gridDim.x * kInsertThreads;
    unsigned int my_new = 0, my_flags = 0;
    for (long long i = (long long)blockIdx.x * kInsertThreads + threadIdx.x; i < n_keys; i += stride) {
        const uint4 a = __ldg(keys + 2 * i), b = __ldg(keys + 2 * i + 1);
        const unsigned long long k[4] = {u64_of(a.x, a.y), u64_of(a.z, a.w), u64_of(b.x, b.y), u64_of(b.z, b.w)};
        if (k[0] == 0ull || k[0] == kClaimed) {
            my_flags |= KVGOV_F_SENTINEL;
            continue;
        }
        switch (insert_one(slots, mask, k, spin_limit)) {
        case kNew: ++my_new; break;
        case kDuplicate: break;
        case kFull: my_flags |= KVGOV_F_TABLE_FULL; break;
        default: my_flags |= KVGOV_F_TIMEOUT; break;
        }
    }
    // Counts: warp reduction, shared-memory accumulation, and the CTA's last
    // warp to finish publishes them (no barrier: early warps just exit).
    const unsigned w_new = __reduce_add_sync(0xffffffffu, my_new);
    const unsigned w_flags = __reduce_or_sync(0xffffffffu, my_flags);
    if ((threadIdx.x & 31) == 0) {
        if (w_new) atomicAdd(&s_new, w_new);
        if (w_flags) atomicOr(&s_flags, w_flags);
        __threadfence_block();
        if (atomicAdd(&s_done, 1u) == kInsertThreads / 32 - 1) {
            const unsigned t_new = atomicAdd(&s_new, 0u), t_flags = atomicOr(&s_flags, 0u);
            if (t_new && n_new) atomicAdd(n_new, (unsigned long long)t_new);
            if (t_flags) atomicOr(status, t_flags);
        }
    }
}

// ---------------------------------------------------------------------------
constexpr int kProbeThreads = 256;

// Is the 32-byte key q in the table?  Reads slots through the read-only path:
// the table does not change during a probe.
__device__ __forceinline__ bool lookup(const uint4 *__restrict__ slots, unsigned long long mask, uint4 q0, uint4 q1) {
    const unsigned long long k0 = u64_of(q0.x, q0.y);
    if (k0 == 0ull || k0 == kClaimed) return false;   // such keys are never stored
    unsigned long long pos = k0 & mask;
    for (unsigned long long n = 0; n <= mask; ++n, pos = (pos + 1) & mask) {
        const uint4 a = __ldg(slots + 2 * pos);
        const unsigned long long w0 = u64_of(a.x, a.y);
        if (w0 == 0ull) return false;
        if (w0 == k0 && a.z == q0.z && a.w == q0.w) {
            const uint4 b = __ldg(slots + 2 * pos + 1);
            if (b.x == q1.x && b.y == q1.y && b.z == q1.z && b.w == q1.w) return true;
        }
    }
    return false;
}

template <int G>
__global__ void __launch_bounds__(kProbeThreads) probe_kernel(const uint4 *__restrict__ slots, unsigned long long mask,
                                                              const uint4 *__restrict__ digests,
                                                              const int64_t *__restrict__ blk_off, int32_t n_req,
                                                              int32_t *__restrict__ prefix_blocks, uint32_t *status) {
    constexpr int kSegs = 32 / G;
    constexpr unsigned kSegMask = G == 32 ? 0xffffffffu : ((1u << G) - 1u);
    const int lane = threadIdx.x & 31, seg = lane / G, sl = lane % G;
    const long long warps_total = (long long)gridDim.x * (kProbeThreads / 32);
    for (long long wg = ((long long)blockIdx.x * kProbeThreads + threadIdx.x) / 32; wg * kSegs < n_req;
         wg += warps_total) {
        const long long r = wg * kSegs + seg;
        long long base = 0, nb = 0;
        bool active = false;
        if (r < n_req) {
            base = blk_off[r];
            nb = blk_off[r + 1] - base;
            if (nb < 0 || base < 0 || base + nb > blk_off[n_req]) {
                if (sl == 0) raise_flag(status, KVGOV_F_BADINDEX);
                nb = 0;
            }
            active = nb > 0;
        }
        long long L = 0;
        const int win = G;
        while (__any_sync(0xffffffffu, active)) {
            const long long j = L + sl;
            const bool mine = active && sl < win && j < nb;
            bool miss = false;
            if (mine) {
                const uint4 *q = digests + 2 * (base + j);
                miss = !lookup(slots, mask, __ldg(q), __ldg(q + 1));
            }
            const unsigned seg_miss = (__ballot_sync(0xffffffffu, miss) >> (seg * G)) & kSegMask;
            if (active) {
                if (seg_miss) {
                    L += __ffs((int)seg_miss) - 1;
                    active = false;
                } else {
                    L += (nb - L < win) ? (nb - L) : win;
                    if (L >= nb) active = false;
                }
            }
        }
        if (r < n_req && sl == 0) prefix_blocks[r] = (int32_t)L;
    }
}

}  // namespace

extern "C" int kvgov_table_init(uint8_t *d_slots, uint64_t capacity, kvgov_stream_t stream) {
    if (!d_slots || !kvgov_host::aligned16(d_slots) || !kvgov_host::pow2_capacity(capacity)) return KVGOV_EINVAL;
    const unsigned long long n_vec = capacity * 2ull;
    unsigned long long grid = (n_vec + 255) / 256;
    if (grid > 152ull * 64) grid = 152ull * 64;
    table_init_kernel<<<(unsigned)grid, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<uint4 *>(d_slots), n_vec);
    return kvgov_host::launch_status();
}

extern "C" int kvgov_insert(uint8_t *d_slots, uint64_t capacity, const uint8_t *d_keys, int64_t n_keys,
                            unsigned long long *d_n_new, uint32_t *d_status, kvgov_stream_t stream) {
    using kvgov_host::aligned16;
    if (!d_slots || !aligned16(d_slots) || !kvgov_host::pow2_capacity(capacity) || n_keys < 0 || !d_status)
        return KVGOV_EINVAL;
    if (n_keys == 0) return KVGOV_OK;
    if (!d_keys || !aligned16(d_keys)) return KVGOV_EINVAL;
    long long grid = (n_keys + kInsertThreads - 1) / kInsertThreads;
    if (grid > 152ll * 64) grid = 152ll * 64;
    insert_kernel<<<(unsigned)grid, kInsertThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<unsigned long long *>(d_slots), capacity - 1, reinterpret_cast<const uint4 *>(d_keys), n_keys,
        d_n_new, d_status, g_spin_limit.load());
    return kvgov_host::launch_status();
}

extern "C" int kvgov_probe(const uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests,
                           const int64_t *d_blk_off, int32_t n_req, int32_t *d_prefix_blocks, uint32_t *d_status,
                           kvgov_stream_t stream) {
    using kvgov_host::aligned16;
    if (!d_slots || !aligned16(d_slots) || !kvgov_host::pow2_capacity(capacity) || n_req < 0) return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;
    if (!d_digests || !aligned16(d_digests) || !d_blk_off || !d_prefix_blocks) return KVGOV_EINVAL;
    constexpr int G = 8;
    const long long warps = ((long long)n_req + (32 / G) - 1) / (32 / G);
    long long grid = (warps + (kProbeThreads / 32) - 1) / (kProbeThreads / 32);
    if (grid > 152ll * 64) grid = 152ll * 64;
    probe_kernel<G><<<(unsigned)grid, kProbeThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<const uint4 *>(d_slots), capacity - 1, reinterpret_cast<const uint4 *>(d_digests), d_blk_off,
        n_req, d_prefix_blocks, d_status);
    return kvgov_host::launch_status();
}

extern "C" uint32_t kvgov_set_spin_limit(uint32_t limit) {
    return g_spin_limit.exchange(limit == 0 ? kDefaultSpin : limit);
}

extern "C" const char *kvgov_status_string(int status) {
    switch (status) {
    case KVGOV_OK: return "KVGOV_OK";
    case KVGOV_EINVAL: return "KVGOV_EINVAL: invalid argument";
    case KVGOV_ECUDA: return "KVGOV_ECUDA: kernel launch failed";
    case (int)KVGOV_F_BADINDEX: return "KVGOV_F_BADINDEX: index or offset out of range";
    case (int)KVGOV_F_SENTINEL: return "KVGOV_F_SENTINEL: reserved key (first 8 bytes all 0x00 or all 0xFF)";
    case (int)KVGOV_F_TABLE_FULL: return "KVGOV_F_TABLE_FULL: no free slot";
    case (int)KVGOV_F_TIMEOUT: return "KVGOV_F_TIMEOUT: gave up waiting for a claimed slot";
    default: return "KVGOV: unknown status";
    }
}
