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
// Slot encoding: the key verbatim as four little-endian u64 words w0..w3.
// (w0, w1) == 0 marks an empty slot.  Home slot = w0 & (capacity - 1);
// collisions go to the next slot (linear probing, wrapping) within a window
// of min(capacity, KVGOV_PROBE_WINDOW) slots: an insert that finds no free
// slot in its key's window fails (table full), so a lookup can stop at the
// end of the window too.  Every walk is bounded, even in a full table.  Keys with
// (w0, w1) == 0, w2 == 0 or w3 == 0 cannot live in a main slot (the first
// pattern marks empty slots, the other two a key still being written): they
// go to the table's side store after the main slots (kvgov_stash.cuh), so
// every key but the all-zero one is stored.
//
// Insert protocol (one key per thread, no fences): walk the slots.  A plain
// read whose two first-half words are both non-zero is final (the half is
// written once, from zero, so a torn read shows a zero word): another key
// means walk on, the key's own first half means compare the second half.
// Any other slot gets a 128-bit compare-and-swap of (w0, w1) from (0, 0) to
// the key's first half, which either claims an empty slot -- then the thread
// stores w2 and w3 -- or returns the occupant's first half atomically.  If that equals the key's,
// the thread waits, a bounded number of re-reads, until w2 and w3 are both
// non-zero (written), then compares them: equal is a duplicate, different is
// another key with the same first half, and the walk goes on.  Two inserts of
// one key in one batch therefore store it once, and no reader can act on a
// half-written slot.
//
// Insert of a probed batch (kvgov_insert_uncached): only the blocks at and
// after each request's first miss, with the same per-key protocol.
//
// Probe: a request's prefix length is its first block not found.  G lanes
// of a warp serve one request and look up a window of its next blocks in
// parallel; a ballot over the window's misses gives the first miss, else the
// window moves on (probe_seg_kernel).  The layout depends on the batch size:
// batches of many requests share each warp's lanes among 16 requests, one
// lane each for block 0 (most requests of a batch of fresh prompts miss
// there), then the lanes of the requests that ended go to those still going
// (probe_share_kernel); mid-size batches 16 lanes per request, windows of 16
// then 32; few requests a warp each, windows of 32, 64, then 128 blocks, so
// that a long cached prefix takes few rounds.  Lookups past the first miss
// inside a window are wasted: they cost bandwidth but not latency.  In every
// layout each lookup first reads its key's home slot and the next one
// together; the walks that go on past them are finished by the whole warp
// at once (warp_finish_walks), and a walk past a miss already found for its
// request is dropped.
#include <atomic>

#include "kvgov_internal.cuh"
#include "kvgov_insert.cuh"
#include "kvgov_lookup.cuh"

namespace {

using namespace kvgov_dev;

constexpr uint32_t kDefaultSpin = 1u << 23;
std::atomic<uint32_t> g_spin_limit{kDefaultSpin};

// ---------------------------------------------------------------------------
__global__ void table_init_kernel(uint4 *__restrict__ slots, unsigned long long n_vec) {
    for (unsigned long long i = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; i < n_vec;
         i += (unsigned long long)gridDim.x * blockDim.x)
        slots[i] = make_uint4(0u, 0u, 0u, 0u);
}

// ---------------------------------------------------------------------------
constexpr int kInsertThreads = 256;

__global__ void __launch_bounds__(kInsertThreads) insert_kernel(unsigned long long *__restrict__ slots,
                                                                unsigned long long mask,
                                                                const uint4 *__restrict__ keys, long long n_keys,
                                                                unsigned long long *n_new, uint32_t *status,
                                                                uint32_t spin_limit) {
    __shared__ unsigned int s_new, s_flags, s_done;
    if (threadIdx.x == 0) { s_new = 0; s_flags = 0; s_done = 0; }
    __syncthreads();
    const long long stride = (long long)gridDim.x * kInsertThreads;
    const int lane = threadIdx.x & 31;
    unsigned int my_new = 0, my_flags = 0;
    // warp-uniform trip count
    for (long long i0 = (long long)blockIdx.x * kInsertThreads + (threadIdx.x & ~31); i0 < n_keys; i0 += stride) {
        const long long i = i0 + lane;
        unsigned long long k[4] = {0ull, 0ull, 0ull, 0ull};
        bool mine = i < n_keys;
        if (mine) {
            const uint4 a = __ldg(keys + 2 * i), b = __ldg(keys + 2 * i + 1);
            k[0] = u64_of(a.x, a.y); k[1] = u64_of(a.z, a.w); k[2] = u64_of(b.x, b.y); k[3] = u64_of(b.z, b.w);
            if (key_is_zero(k)) {
                my_flags |= KVGOV_F_SENTINEL;
                mine = false;
            }
        }
        if (mine) count_insert(insert_one(slots, mask, k, spin_limit), my_new, my_flags);
    }
    publish_counts(my_new, my_flags, &s_new, &s_flags, &s_done, n_new, status);
}

// ---------------------------------------------------------------------------
constexpr int kProbeThreads = 256;
// Probe layouts by batch size (measured side by side over every workload):
// probe_seg_kernel<G, kPer, PAIR, COOP> with first window F.  PAIR reads a key's
// home slot and the next one together (a walk of two slots in one memory
// round trip) rather than the home slot alone.
// COOP finishes the walks that go past their first slots with the whole
// warp (warp_finish_walks) rather than each lane on its own: it pays where
// the table is loaded and many lanes look up at once (mid-size batches:
// 8.5 -> 6.5 us on 4096 requests at load factor 0.5), not with one request
// a warp, whose four lookups a lane would finish one after another (a
// 2048-block prefix: 45 -> 57 us).
struct ProbeLayout { int min_req, G, per, pair, first, coop; };
constexpr int32_t kProbeShareMin = 32768;               // n_req >= 32768: probe_share_kernel
constexpr int kProbeShareR = 16;                         // ... with 16 requests per warp
constexpr bool kProbeSharePair = true;                   // ... reading the home slot and the next together
constexpr ProbeLayout kProbeMid{2048, 16, 2, 1, 16, 1};    // 2048 <= n_req < 32768
constexpr ProbeLayout kProbeFew{0, 32, 4, 1, 32, 0};     // fewer

// Request r's block range; a malformed one is flagged and counts as empty.
__device__ __forceinline__ void probe_range(const int64_t *__restrict__ blk_off, int32_t n_req, long long r,
                                            long long &base, long long &nb, uint32_t *status) {
    base = blk_off[r];
    nb = blk_off[r + 1] - base;
    if (nb < 0 || base < 0 || base + nb > blk_off[n_req]) {
        raise_flag(status, KVGOV_F_BADINDEX);
        nb = 0;
    }
}

// Where request r's walk starts: block 0, or (resume) the block s its
// prefix_blocks entry names -- a lower bound of its cached prefix, left there
// by lookups that ran while the table was still growing -- clamped to
// [0, nb].  The entry is read beside the request's offsets, not after them.
__device__ __forceinline__ long long probe_start(long long s, long long nb) {
    return s < 0 ? 0 : (s > nb ? nb : s);
}

// G lanes per request (32 / G requests per warp).  A request's first round
// looks up its first `first` blocks; later rounds G, 2G, 4G ... blocks up to
// G * kPer (kPer lookups per lane, their home slots read together so that
// their memory accesses overlap).  A small first window wastes few lookups
// on a request that misses early; the growing windows take a long cached
// prefix in few rounds.
template <int G, int kPer, bool PAIR, bool COOP>
__global__ void __launch_bounds__(kProbeThreads) probe_seg_kernel(const uint4 *__restrict__ slots,
                                                                  unsigned long long mask,
                                                                  const uint4 *__restrict__ digests,
                                                                  const int64_t *__restrict__ blk_off,
                                                                  int32_t n_req, int32_t *prefix_blocks,
                                                                  uint32_t *status, int first, bool resume) {
    constexpr int kSegs = 32 / G;
    constexpr unsigned kSegMask = G == 32 ? 0xffffffffu : ((1u << G) - 1u);
    const int lane = threadIdx.x & 31, seg = lane / G, sl = lane % G;
    const long long warps_total = (long long)gridDim.x * (kProbeThreads / 32);
    for (long long wg = ((long long)blockIdx.x * kProbeThreads + threadIdx.x) / 32; wg * kSegs < n_req;
         wg += warps_total) {                                  // warp-uniform
        const long long r = wg * kSegs + seg;
        long long base = 0, nb = 0, s0 = 0;
        if (r < n_req) {
            if (resume) s0 = prefix_blocks[r];
            probe_range(blk_off, n_req, r, base, nb, sl == 0 ? status : nullptr);
        }
        long long L = probe_start(s0, nb);
        int w = first;
        bool active = nb > L;
        while (__any_sync(0xffffffffu, active)) {
            uint4 q0[kPer], q1[kPer], a[kPer], b[kPer], c[kPer], d[kPer];
#pragma unroll
            for (int u = 0; u < kPer; ++u) {
                const int o = sl + G * u;
                q0[u] = q1[u] = make_uint4(0u, 0u, 0u, 0u);
                if (active && o < w && L + o < nb) {
                    q0[u] = __ldg(digests + 2 * (base + L + o));
                    q1[u] = __ldg(digests + 2 * (base + L + o) + 1);
                }
            }
#pragma unroll
            for (int u = 0; u < kPer; ++u) {
                const int o = sl + G * u;
                if (active && o < w && L + o < nb) {
                    const unsigned long long h = home_slot(q0[u], mask);
                    a[u] = __ldg(slots + 2 * h);
                    b[u] = __ldg(slots + 2 * h + 1);
                    c[u] = a[u];
                    d[u] = b[u];
                    if (PAIR) {
                        const unsigned long long h1 = (h + 1) & mask;
                        c[u] = __ldg(slots + 2 * h1);
                        d[u] = __ldg(slots + 2 * h1 + 1);
                    }
                }
            }
            int miss_at = -1;                                  // the window's first miss (per segment)
#pragma unroll
            for (int u = 0; u < kPer; ++u) {
                const int o = sl + G * u;
                const bool valid = active && o < w && L + o < nb;
                int st = valid ? walk_start<PAIR ? 2 : 1>(slots, mask, q0[u], q1[u], a[u], b[u], c[u], d[u]) : 1;
                if (COOP) {
                    // a walk past a miss already found for its request decides nothing: drop it
                    const unsigned m0 = (__ballot_sync(0xffffffffu, st == 0) >> (seg * G)) & kSegMask;
                    if (st < 0 && (miss_at >= 0 || (m0 & ((1u << sl) - 1u)))) st = 0;
                    st = warp_finish_walks<PAIR ? 2 : 1>(slots, mask, q0[u], q1[u], st);
                } else if (st < 0) {
                    st = walk_on<PAIR ? 2 : 1>(slots, mask, q0[u], q1[u]);
                }
                const unsigned m = (__ballot_sync(0xffffffffu, valid && st == 0) >> (seg * G)) & kSegMask;
                if (m && miss_at < 0) miss_at = G * u + __ffs((int)m) - 1;
            }
            if (active) {
                if (miss_at >= 0) {
                    L += miss_at;
                    active = false;
                } else {
                    L += (nb - L < w) ? (nb - L) : w;
                    if (L >= nb) active = false;
                }
                w = w < G ? G : (2 * w < G * kPer ? 2 * w : G * kPer);
            }
        }
        if (r < n_req && sl == 0) prefix_blocks[r] = (int32_t)L;
    }
}

// Large batches: R requests per warp, and in each round the warp's 32 lanes
// are shared out among the requests still active -- 32 / k consecutive lanes
// each when k are active -- every lane looking up one block (its home slot
// and the next, read together).  The first round gives each request one lane
// (block 0: most requests of a batch of fresh prompts miss there); then a
// request that goes on gets the lanes of those that ended, so a long cached
// prefix takes few rounds however short its warp-mates' are.  Request state
// (row base, block count, prefix so far) stays in lanes 0..R-1 and is
// shuffled to the lanes that serve it.
template <int R, bool PAIR>
__global__ void __launch_bounds__(kProbeThreads) probe_share_kernel(const uint4 *__restrict__ slots,
                                                                    unsigned long long mask,
                                                                    const uint4 *__restrict__ digests,
                                                                    const int64_t *__restrict__ blk_off,
                                                                    int32_t n_req, int32_t *prefix_blocks,
                                                                    uint32_t *status, bool resume) {
    constexpr unsigned kReqMask = (1u << R) - 1u;
    const int lane = threadIdx.x & 31;
    const long long warps_total = (long long)gridDim.x * (kProbeThreads / 32);
    for (long long wg = ((long long)blockIdx.x * kProbeThreads + threadIdx.x) / 32; wg * R < n_req;
         wg += warps_total) {                                  // warp-uniform
        const long long r = wg * R + lane;                     // lanes 0..R-1: request r
        long long base = 0, nb = 0, L = 0;
        if (lane < R && r < n_req) {
            const long long s0 = resume ? prefix_blocks[r] : 0;
            probe_range(blk_off, n_req, r, base, nb, status);
            L = probe_start(s0, nb);
        }
        unsigned act = __ballot_sync(0xffffffffu, lane < R && nb > L) & kReqMask;
        bool first = true;
        while (act) {                                          // warp-uniform
            const int k = __popc(act);
            const int lp = first ? 1 : 32 / k;                 // lanes per active request this round
            const int rho = lane / lp, o = lane % lp;          // the active request this lane serves, its block
            const int s = rho < k ? __fns(act, 0, rho + 1) : 0;
            const long long sb = __shfl_sync(0xffffffffu, base, s);
            const long long snb = __shfl_sync(0xffffffffu, nb, s);
            const long long sL = __shfl_sync(0xffffffffu, L, s);
            const bool valid = rho < k && sL + o < snb;
            uint4 q0 = make_uint4(0u, 0u, 0u, 0u), q1 = q0;
            int st = 1;                                        // walk state (walk_start); no lookup: not a miss
            if (valid) {
                q0 = __ldg(digests + 2 * (sb + sL + o));
                q1 = __ldg(digests + 2 * (sb + sL + o) + 1);
                const unsigned long long h = home_slot(q0, mask);
                const uint4 a = __ldg(slots + 2 * h), b = __ldg(slots + 2 * h + 1);
                uint4 c = a, d = b;
                if (PAIR) {
                    const unsigned long long h1 = (h + 1) & mask;
                    c = __ldg(slots + 2 * h1);
                    d = __ldg(slots + 2 * h1 + 1);
                }
                st = walk_start<PAIR ? 2 : 1>(slots, mask, q0, q1, a, b, c, d);
            }
            {   // a walk past a miss already found for its request decides nothing: drop it
                const unsigned m0 = __ballot_sync(0xffffffffu, st == 0);
                const unsigned grp = lp == 32 ? 0xffffffffu : ((1u << lp) - 1u) << (rho * lp);
                if (st < 0 && (m0 & grp & ((1u << lane) - 1u))) st = 0;
            }
            st = warp_finish_walks<PAIR ? 2 : 1>(slots, mask, q0, q1, st);
            const bool miss = valid && st == 0;
            const unsigned mb = __ballot_sync(0xffffffffu, miss);
            if (lane < R && ((act >> lane) & 1u)) {
                const int my = __popc(act & ((1u << lane) - 1u));       // this request's rank among the active
                const unsigned seg = (mb >> (my * lp)) & (lp == 32 ? 0xffffffffu : ((1u << lp) - 1u));
                if (seg) {
                    L += __ffs((int)seg) - 1;
                    act &= ~(1u << lane);
                } else {
                    L += (nb - L < lp) ? (nb - L) : lp;
                    if (L >= nb) act &= ~(1u << lane);
                }
            }
            act = __ballot_sync(0xffffffffu, lane < R && ((act >> lane) & 1u)) & kReqMask;
            first = false;
        }
        if (lane < R && r < n_req) prefix_blocks[r] = (int32_t)L;
    }
}

// Insert every request's blocks from its cached-prefix length on (the output
// of kvgov_probe): the blocks before it were found in the table, and a table
// only grows, so inserting them would change nothing.  The uncached blocks
// of kPackReq requests are packed into the 32 lanes of a warp: lanes 0..kPackReq-1 read their request's range and
// count of uncached blocks, a warp scan numbers the blocks, and in each round
// lane l takes block i0 + l, finding its request with a 5-step search over the
// scan.  No lane idles while blocks remain (with 8 lanes per request, a
// request with 4 cached and 4 uncached blocks leaves half the lanes idle;
// measured faster than that layout).
constexpr int kPackReq = 8;

__global__ void __launch_bounds__(kInsertThreads) insert_uncached_packed_kernel(
    unsigned long long *__restrict__ slots, unsigned long long mask, const uint4 *__restrict__ digests,
    const int64_t *__restrict__ blk_off, int32_t n_req, const int32_t *__restrict__ prefix_blocks,
    unsigned long long *n_new, uint32_t *status, uint32_t spin_limit, uint32_t *gen, uint32_t g) {
    // gen: nullable; a slot (or side-store entry) this launch claims gets generation g
    __shared__ unsigned int s_new, s_flags, s_done;
    if (threadIdx.x == 0) { s_new = 0; s_flags = 0; s_done = 0; }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const long long warps_total = (long long)gridDim.x * (kInsertThreads / 32);
    unsigned my_new = 0, my_flags = 0;
    for (long long w = ((long long)blockIdx.x * kInsertThreads + threadIdx.x) / 32; w * kPackReq < n_req;
         w += warps_total) {                                   // warp-uniform
        const long long r = w * kPackReq + lane;
        long long first = 0;                                   // row of the request's first uncached block
        int c = 0;                                             // its uncached blocks
        if (lane < kPackReq && r < n_req) {
            const long long base = blk_off[r], nb = blk_off[r + 1] - base;
            if (nb < 0 || base < 0 || base + nb > blk_off[n_req]) {
                my_flags |= KVGOV_F_BADINDEX;
            } else {
                long long L = prefix_blocks[r];
                L = L < 0 ? 0 : (L > nb ? nb : L);
                first = base + L;
                c = (int)(nb - L);
            }
        }
        int incl = c;                                          // inclusive scan of c over the lanes
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, incl, d);
            if (lane >= d) incl += t;
        }
        const int total = __shfl_sync(0xffffffffu, incl, 31);
        for (int i0 = 0; i0 < total; i0 += 32) {               // warp-uniform
            const int k = i0 + lane;
            int lo = 0, hi = 31;                               // the first lane whose scan passes k
#pragma unroll
            for (int step = 0; step < 5; ++step) {
                const int mid = (lo + hi) >> 1;
                if (__shfl_sync(0xffffffffu, incl, mid) > k) hi = mid;
                else lo = mid + 1;
            }
            const long long f = __shfl_sync(0xffffffffu, first, lo);
            const int before = __shfl_sync(0xffffffffu, incl - c, lo);
            bool mine = k < total;
            unsigned long long key[4] = {0ull, 0ull, 0ull, 0ull};
            if (mine) {
                const long long row = f + (k - before);
                const uint4 a = __ldg(digests + 2 * row), b = __ldg(digests + 2 * row + 1);
                key[0] = u64_of(a.x, a.y); key[1] = u64_of(a.z, a.w);
                key[2] = u64_of(b.x, b.y); key[3] = u64_of(b.z, b.w);
                if (key_is_zero(key)) {
                    my_flags |= KVGOV_F_SENTINEL;
                    mine = false;
                }
            }
            if (mine) {
                unsigned long long pos = 0;
                const InsertResult res = insert_one(slots, mask, key, spin_limit, &pos);
                count_insert(res, my_new, my_flags);
                if (gen && res == kNew) gen[pos] = g;
            }
        }
    }
    publish_counts(my_new, my_flags, &s_new, &s_flags, &s_done, n_new, status);
}

// G lanes per request: 32 / G requests per warp, at most 64 CTAs per SM.
unsigned probe_grid(int32_t n_req, int G) {
    const long long per_warp = 32 / G;
    const long long warps = ((long long)n_req + per_warp - 1) / per_warp;
    long long grid = (warps + (kProbeThreads / 32) - 1) / (kProbeThreads / 32);
    const long long cap = (long long)kvgov_host::sm_count() * 64;
    return (unsigned)(grid < cap ? grid : cap);
}

}  // namespace

extern "C" int kvgov_table_init(uint8_t *d_slots, uint64_t capacity, kvgov_stream_t stream) {
    if (!d_slots || !kvgov_host::aligned16(d_slots) || !kvgov_host::pow2_capacity(capacity)) return KVGOV_EINVAL;
    const unsigned long long n_vec = (capacity + KVGOV_STASH_SLOTS) * 2ull;   // main slots and side store
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

namespace {

// kvgov_probe, or (resume) its walks continued from each request's
// prefix_blocks entry (kvgov_host::probe_resume).
int launch_probe(const uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests, const int64_t *d_blk_off,
                 int32_t n_req, int32_t *d_prefix_blocks, uint32_t *d_status, kvgov_stream_t stream, bool resume) {
    using kvgov_host::aligned16;
    if (!d_slots || !aligned16(d_slots) || !kvgov_host::pow2_capacity(capacity) || n_req < 0) return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;
    if (!d_digests || !aligned16(d_digests) || !d_blk_off || !d_prefix_blocks) return KVGOV_EINVAL;
    const uint4 *slots = reinterpret_cast<const uint4 *>(d_slots), *dig = reinterpret_cast<const uint4 *>(d_digests);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (n_req >= kProbeShareMin)
        probe_share_kernel<kProbeShareR, kProbeSharePair><<<probe_grid(n_req, 32 / kProbeShareR), kProbeThreads, 0, s>>>(
            slots, capacity - 1, dig, d_blk_off, n_req, d_prefix_blocks, d_status, resume);
    else if (n_req >= kProbeMid.min_req)
        probe_seg_kernel<kProbeMid.G, kProbeMid.per, kProbeMid.pair != 0, kProbeMid.coop != 0>
            <<<probe_grid(n_req, kProbeMid.G), kProbeThreads, 0, s>>>(
                slots, capacity - 1, dig, d_blk_off, n_req, d_prefix_blocks, d_status, kProbeMid.first, resume);
    else
        probe_seg_kernel<kProbeFew.G, kProbeFew.per, kProbeFew.pair != 0, kProbeFew.coop != 0>
            <<<probe_grid(n_req, kProbeFew.G), kProbeThreads, 0, s>>>(
                slots, capacity - 1, dig, d_blk_off, n_req, d_prefix_blocks, d_status, kProbeFew.first, resume);
    return kvgov_host::launch_status();
}

}  // namespace

namespace kvgov_host {
int probe_resume(const uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests, const int64_t *d_blk_off,
                 int32_t n_req, int32_t *d_prefix_blocks, uint32_t *d_status, kvgov_stream_t stream) {
    return launch_probe(d_slots, capacity, d_digests, d_blk_off, n_req, d_prefix_blocks, d_status, stream, true);
}
}  // namespace kvgov_host

extern "C" int kvgov_probe_resume(const uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests,
                                  const int64_t *d_blk_off, int32_t n_req, int32_t *d_prefix_blocks,
                                  uint32_t *d_status, kvgov_stream_t stream) {
    return kvgov_host::probe_resume(d_slots, capacity, d_digests, d_blk_off, n_req, d_prefix_blocks, d_status,
                                    stream);
}

extern "C" int kvgov_probe(const uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests,
                           const int64_t *d_blk_off, int32_t n_req, int32_t *d_prefix_blocks, uint32_t *d_status,
                           kvgov_stream_t stream) {
    return launch_probe(d_slots, capacity, d_digests, d_blk_off, n_req, d_prefix_blocks, d_status, stream, false);
}

extern "C" int kvgov_insert_uncached(uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests,
                                     const int64_t *d_blk_off, int32_t n_req, const int32_t *d_prefix_blocks,
                                     unsigned long long *d_n_new, uint32_t *d_status, kvgov_stream_t stream) {
    return kvgov_host::insert_uncached_gen(d_slots, capacity, d_digests, d_blk_off, n_req, d_prefix_blocks, d_n_new,
                                           d_status, nullptr, 0, stream);
}

// kvgov_insert_uncached, a slot it claims getting generation `gen` when
// d_gen is given (kvgov_chain_hash_serve's small-batch path).
int kvgov_host::insert_uncached_gen(uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests,
                                    const int64_t *d_blk_off, int32_t n_req, const int32_t *d_prefix_blocks,
                                    unsigned long long *d_n_new, uint32_t *d_status, uint32_t *d_gen, uint32_t gen,
                                    kvgov_stream_t stream) {
    using kvgov_host::aligned16;
    if (!d_slots || !aligned16(d_slots) || !kvgov_host::pow2_capacity(capacity) || n_req < 0 || !d_status)
        return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;
    if (!d_digests || !aligned16(d_digests) || !d_blk_off || !d_prefix_blocks) return KVGOV_EINVAL;
    const long long warps = ((long long)n_req + kPackReq - 1) / kPackReq;
    long long grid = (warps + (kInsertThreads / 32) - 1) / (kInsertThreads / 32);
    if (grid > 152ll * 64) grid = 152ll * 64;
    insert_uncached_packed_kernel<<<(unsigned)grid, kInsertThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<unsigned long long *>(d_slots), capacity - 1, reinterpret_cast<const uint4 *>(d_digests),
        d_blk_off, n_req, d_prefix_blocks, d_n_new, d_status, g_spin_limit.load(), d_gen, gen);
    return kvgov_host::launch_status();
}

namespace {

// gen[h] = value for every handle h that holds a key (main slots whose first
// half is not zero, live side-store entries), 0 for every other.
__global__ void gen_stamp_kernel(const uint4 *__restrict__ slots, unsigned long long capacity,
                                 uint32_t *__restrict__ gen, uint32_t value) {
    const unsigned long long n = capacity + KVGOV_STASH_SLOTS;
    const uint32_t *state = reinterpret_cast<const uint32_t *>(slots + 2 * capacity) + 8;
    const uint32_t handed = *reinterpret_cast<const uint32_t *>(slots + 2 * capacity);
    for (unsigned long long h = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; h < n;
         h += (unsigned long long)gridDim.x * blockDim.x) {
        bool held;
        if (h < capacity) {
            const uint4 a = slots[2 * h];
            held = (a.x | a.y | a.z | a.w) != 0u;
        } else {
            const long long e = (long long)(h - capacity) - kStashHeaderSlots;   // side-store entry
            held = e >= 0 && e < (long long)handed && e < KVGOV_STASH_KEYS && state[e] == kStashLive;
        }
        gen[h] = held ? value : 0u;
    }
}

}  // namespace

extern "C" int kvgov_table_gen_stamp(const uint8_t *d_slots, uint64_t capacity, uint32_t *d_gen, uint32_t value,
                                     kvgov_stream_t stream) {
    if (!d_slots || !kvgov_host::aligned16(d_slots) || !kvgov_host::pow2_capacity(capacity) || !d_gen)
        return KVGOV_EINVAL;
    unsigned long long grid = (capacity + KVGOV_STASH_SLOTS + 255) / 256;
    if (grid > 152ull * 64) grid = 152ull * 64;
    gen_stamp_kernel<<<(unsigned)grid, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<const uint4 *>(d_slots), capacity, d_gen, value);
    return kvgov_host::launch_status();
}

namespace kvgov_host {
uint32_t spin_limit() { return g_spin_limit.load(); }
}  // namespace kvgov_host

extern "C" uint32_t kvgov_set_spin_limit(uint32_t limit) {
    return g_spin_limit.exchange(limit == 0 ? kDefaultSpin : limit);
}

extern "C" const char *kvgov_status_string(int status) {
    switch (status) {
    case KVGOV_OK: return "KVGOV_OK";
    case KVGOV_EINVAL: return "KVGOV_EINVAL: invalid argument";
    case KVGOV_ECUDA: return "KVGOV_ECUDA: kernel launch failed";
    case (int)KVGOV_F_BADINDEX: return "KVGOV_F_BADINDEX: index or offset out of range";
    case (int)KVGOV_F_SENTINEL: return "KVGOV_F_SENTINEL: the all-zero key (an empty slot's value) was not stored";
    case (int)KVGOV_F_TABLE_FULL: return "KVGOV_F_TABLE_FULL: no free slot in a key's window or the side store";
    case (int)KVGOV_F_TIMEOUT: return "KVGOV_F_TIMEOUT: gave up waiting for a slot's key to be written";
    default: return "KVGOV: unknown status";
    }
}
