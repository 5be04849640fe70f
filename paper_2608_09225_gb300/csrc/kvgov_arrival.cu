// kvgov_arrival.cu -- arrival-order serving of one batch (kvgov_owner_init,
// kvgov_insert_arrival, kvgov_probe_arrival).
//
// Paper: section 2.1 (a lookup matches the longest cached prefix of blocks
// from position 0; any request sharing the prefix hits the same blocks) and
// section 4.2 (prefill cost is proportional to the uncached tokens).  A
// serving cache meets the requests of a batch one after another: request r
// finds the blocks that were cached before the batch and those of every
// request that arrived before it, and after its prefill all its blocks are
// cached.  Served one request at a time that is a probe and an insert per
// request; here the whole batch is served in three launches that give the
// same prefix lengths.
//
// Every slot of the table has an owner (u64, in a caller-owned array beside
// the slots): the smallest arrival position of a block that inserted the
// slot's key through kvgov_insert_arrival, or 0 -- before every arrival -- for
// a key inserted any other way.  Blocks arrive in request-major order: block
// j of request r has position seq_base + blk_off[r] + j, so a key first seen
// in an earlier request has a smaller position than every block of r.
//
//   insert_arrival_kernel  one thread per block: inserts its key (the insert
//                          protocol of kvgov_table.cu) and records the slot
//                          that holds it in slot_of.  A block whose insert
//                          claims a slot (a key new to the table) writes its own
//                          position as the owner -- no other thread writes that
//                          owner in this launch -- and marks its slot_of entry
//                          settled.
//   owner_min_kernel       after every claim, one thread per block: for each
//                          block not marked, an atomic min of its slot's owner
//                          with its position, which can only lower an owner
//                          set in this batch (any other owner belongs to an
//                          earlier batch or to no arrival, so it is smaller);
//                          owners end at the first block that holds their key.
//                          The marks are cleared.
//   probe_arrival_kernel   after every min: block j of request r was cached
//                          when r arrived iff its slot's owner is below the
//                          position of r's first block.  The prefix ends at the
//                          first block that was not (or whose key could not be
//                          stored).
//
// A key held in the table's side store (kvgov_stash.cuh) has the handle
// capacity + 8 + its entry, so the owner array has capacity +
// KVGOV_STASH_SLOTS entries.
#include <atomic>

#include "kvgov_insert.cuh"
#include "kvgov_internal.cuh"

namespace {

using namespace kvgov_dev;

// Largest first position of a batch (positions stay below 2^63 for any batch
// that fits in memory).
constexpr unsigned long long kMaxSeq = 1ull << 62;
constexpr long long kNoRowCap = 0x7fffffffffffffffll;   // slot_of sized by the caller
constexpr int kThreads = 256;
constexpr int G = 8;                         // lanes per request
constexpr int kSegs = 32 / G;
constexpr unsigned kSegMask = (1u << G) - 1u;

__global__ void owner_init_kernel(uint4 *__restrict__ owner, unsigned long long n_vec) {
    for (unsigned long long i = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; i < n_vec;
         i += (unsigned long long)gridDim.x * blockDim.x)
        owner[i] = make_uint4(0u, 0u, 0u, 0u);
}

// Request r and its block range, with the same validity check as the probe:
// a malformed range flags KVGOV_F_BADINDEX and counts as empty.
__device__ __forceinline__ void request_range(const int64_t *__restrict__ blk_off, int32_t n_req, long long r,
                                              long long &base, long long &nb, unsigned &flags) {
    base = 0;
    nb = 0;
    if (r >= n_req) return;
    base = blk_off[r];
    nb = blk_off[r + 1] - base;
    if (nb < 0 || base < 0 || base + nb > blk_off[n_req]) {
        flags |= KVGOV_F_BADINDEX;
        nb = 0;
    }
}

// The batch's block count, blk_off[n_req] (0, flagged, if negative or above
// row_cap, the rows slot_of can hold).
__device__ __forceinline__ long long batch_rows(const int64_t *__restrict__ blk_off, int32_t n_req, uint32_t *status,
                                                bool flag, long long row_cap) {
    const long long n = blk_off[n_req];
    if (n < 0 || n > row_cap) {
        if (flag && blockIdx.x == 0 && threadIdx.x == 0) raise_flag(status, KVGOV_F_BADINDEX);
        return 0;
    }
    return n;
}

__global__ void __launch_bounds__(kThreads) insert_arrival_kernel(
    unsigned long long *__restrict__ slots, unsigned long long mask, unsigned long long *__restrict__ owner,
    const uint4 *__restrict__ digests, const int64_t *__restrict__ blk_off, int32_t n_req,
    uint32_t *__restrict__ slot_of, unsigned long long *n_new, uint32_t *status, uint32_t spin_limit,
    long long row_cap, unsigned long long seq_base, int32_t first_req) {
    __shared__ unsigned int s_new, s_flags, s_done;
    if (threadIdx.x == 0) { s_new = 0; s_flags = 0; s_done = 0; }
    __syncthreads();
    long long n_rows = batch_rows(blk_off, n_req, status, first_req == 0, row_cap);
    // first_req > 0: only the blocks of requests [0, first_req), and no slot handles
    if (first_req > 0 && n_rows > 0) {
        const long long lim = blk_off[first_req];
        n_rows = lim < 0 ? 0 : (lim < n_rows ? lim : n_rows);
    }
    const bool handles = first_req == 0;
    const long long stride = (long long)gridDim.x * kThreads;
    const int lane = threadIdx.x & 31;
    unsigned my_new = 0, my_flags = 0;
    for (long long i0 = (long long)blockIdx.x * kThreads + (threadIdx.x & ~31); i0 < n_rows; i0 += stride) {
        const long long row = i0 + lane;                       // warp-uniform trip count
        if (row >= n_rows) continue;
        const uint4 a = __ldg(digests + 2 * row), b = __ldg(digests + 2 * row + 1);
        const unsigned long long k[4] = {u64_of(a.x, a.y), u64_of(a.z, a.w), u64_of(b.x, b.y), u64_of(b.z, b.w)};
        if (key_is_zero(k)) {
            if (handles) {
                my_flags |= KVGOV_F_SENTINEL;
                slot_of[row] = kNoSlot;
            }
            continue;
        }
        unsigned long long pos = 0;
        const InsertResult res = insert_one(slots, mask, k, spin_limit, &pos);
        count_insert(res, my_new, my_flags);
        if (res == kNew) owner[pos] = seq_base + (unsigned long long)row;   // settled: the first writer's position
        if (handles)
            slot_of[row] = res == kNew ? ((uint32_t)pos | kSettled) : (res == kDuplicate ? (uint32_t)pos : kNoSlot);
    }
    publish_counts(my_new, my_flags, &s_new, &s_flags, &s_done, n_new, status);
}

__global__ void __launch_bounds__(kThreads) owner_min_kernel(const int64_t *__restrict__ blk_off, int32_t n_req,
                                                             uint32_t *__restrict__ slot_of,
                                                             unsigned long long *__restrict__ owner,
                                                             unsigned long long seq_base, long long row_cap) {
    const long long n_rows = batch_rows(blk_off, n_req, nullptr, false, row_cap);
    const long long stride = (long long)gridDim.x * kThreads;
    const int lane = threadIdx.x & 31;
    for (long long r0 = (long long)blockIdx.x * kThreads + (threadIdx.x & ~31); r0 < n_rows; r0 += stride) {
        const long long row = r0 + lane;                       // warp-uniform trip count
        uint32_t s = row < n_rows ? slot_of[row] : kNoSlot;
        if (s != kNoSlot && (s & kSettled)) {                  // settled by the insert: clear the mark
            slot_of[row] = s & ~kSettled;
            s = kNoSlot;
        }
        // Shared prefixes put one key in many rows: within a warp only the
        // lowest row of each slot takes part (rows ascend with the lane), and
        // it skips the atomic when the owner already holds an earlier
        // position (owners only decrease while this kernel runs).
        const unsigned same = __match_any_sync(0xffffffffu, s);
        if (s == kNoSlot || lane != __ffs(same) - 1) continue;
        const unsigned long long p = seq_base + (unsigned long long)row;
        if (ld_relaxed(owner + s) > p) atomicMin(owner + s, p);
    }
}

// The same min with one thread per request walking its blocks, for batches
// of many requests (after the fused chain insert): the 32 lanes of a warp
// hold block j of 32 consecutive requests, so one key shared by their
// prefixes is settled once per warp.  Eight blocks at a time: their slot
// handles, then the owners of the slots this lane settles, then the atomics,
// so that each group of eight costs two memory round trips rather than
// sixteen.
__global__ void __launch_bounds__(kThreads) owner_min_req_kernel(const int64_t *__restrict__ blk_off, int32_t n_req,
                                                                 uint32_t *__restrict__ slot_of,
                                                                 unsigned long long *__restrict__ owner,
                                                                 unsigned long long seq_base) {
    constexpr int kGroup = 8;
    const long long r = (long long)blockIdx.x * kThreads + threadIdx.x;
    const int lane = threadIdx.x & 31;
    long long base, nb;
    unsigned ignored = 0;                         // the insert has flagged bad ranges
    request_range(blk_off, n_req, r, base, nb, ignored);
    const int jmax = __reduce_max_sync(0xffffffffu, (unsigned)nb);
    for (int j0 = 0; j0 < jmax; j0 += kGroup) {                // warp-uniform
        uint32_t s[kGroup];
#pragma unroll
        for (int u = 0; u < kGroup; ++u) {
            s[u] = j0 + u < nb ? slot_of[base + j0 + u] : kNoSlot;
            if (s[u] != kNoSlot && (s[u] & kSettled)) {        // settled by the insert: clear the mark
                slot_of[base + j0 + u] = s[u] & ~kSettled;
                s[u] = kNoSlot;
            }
        }
        bool lead[kGroup];
#pragma unroll
        for (int u = 0; u < kGroup; ++u) {
            const unsigned same = __match_any_sync(0xffffffffu, s[u]);
            lead[u] = s[u] != kNoSlot && lane == __ffs(same) - 1;   // the lowest lane: the earliest position
        }
        unsigned long long cur[kGroup];
#pragma unroll
        for (int u = 0; u < kGroup; ++u) cur[u] = lead[u] ? ld_relaxed(owner + s[u]) : 0ull;
#pragma unroll
        for (int u = 0; u < kGroup; ++u) {
            const unsigned long long p = seq_base + (unsigned long long)(base + j0 + u);
            if (lead[u] && cur[u] > p) atomicMin(owner + s[u], p);
        }
    }
}

__global__ void __launch_bounds__(kThreads) probe_arrival_kernel(const unsigned long long *__restrict__ owner,
                                                                 const uint32_t *__restrict__ slot_of,
                                                                 const int64_t *__restrict__ blk_off, int32_t n_req,
                                                                 unsigned long long seq_base,
                                                                 int32_t *__restrict__ prefix_blocks, uint32_t *status,
                                                                 long long row_cap) {
    const int lane = threadIdx.x & 31, seg = lane / G, sl = lane % G;
    const long long warps_total = (long long)gridDim.x * (kThreads / 32);
    const bool over = blk_off[n_req] > row_cap;           // the insert stored no slot: every request is bad
    for (long long w = ((long long)blockIdx.x * kThreads + threadIdx.x) / 32; w * kSegs < n_req;
         w += warps_total) {                                   // warp-uniform
        const long long r = w * kSegs + seg;
        long long base, nb;
        unsigned flags = 0;
        request_range(blk_off, n_req, r, base, nb, flags);
        if (over && r < n_req) {
            flags |= KVGOV_F_BADINDEX;
            nb = 0;
        }
        if (flags && sl == 0) raise_flag(status, flags);
        const unsigned long long first = seq_base + (unsigned long long)base;   // position of r's block 0
        bool active = nb > 0;
        long long L = 0;
        while (__any_sync(0xffffffffu, active)) {
            const long long j = L + sl;
            bool miss = false;
            if (active && j < nb) {
                const uint32_t s = __ldg(slot_of + base + j);
                miss = s == kNoSlot || __ldg(owner + s) >= first;
            }
            const unsigned seg_miss = (__ballot_sync(0xffffffffu, miss) >> (seg * G)) & kSegMask;
            if (active) {
                if (seg_miss) {
                    L += __ffs((int)seg_miss) - 1;
                    active = false;
                } else {
                    L += (nb - L < G) ? (nb - L) : G;
                    if (L >= nb) active = false;
                }
            }
        }
        if (r < n_req && sl == 0) prefix_blocks[r] = (int32_t)L;
    }
}

// Per-request kernel: G lanes per request, at most 64 CTAs of 256 threads per SM.
unsigned request_grid(int32_t n_req) {
    const long long warps = ((long long)n_req + kSegs - 1) / kSegs;
    long long grid = (warps + (kThreads / 32) - 1) / (kThreads / 32);
    const long long cap = (long long)kvgov_host::sm_count() * 64;
    if (grid > cap) grid = cap;
    return grid < 1 ? 1u : (unsigned)grid;
}

// Per-block kernels: the block count is on the device, so a fixed grid of 8
// resident CTAs per SM strides over the blocks.
unsigned row_grid() { return (unsigned)(kvgov_host::sm_count() * 8); }

// Capacities whose slot index fits slot_of's u32 below the kSettled mark.
bool arrival_capacity(uint64_t capacity) {
    return kvgov_host::pow2_capacity(capacity) && capacity <= (1ull << 30);
}

// Scratch of kvgov_serve_arrival_static: the slot of each block of one batch,
// 2^21 entries (8 MiB), in a file-scope device array instead of caller
// memory.  Every call on the device uses it, so calls must not overlap.
constexpr long long kStaticRows = 1ll << 21;
static __device__ __align__(256) uint32_t g_static_slot_of[kStaticRows];

// Its device address on the current device, looked up with
// cudaGetSymbolAddress on the first call made with that device current and
// kept for the life of the process.  Host threads that make their first calls
// at the same time may each look it up; they store the same address.
uint32_t *static_slot_of() {
    constexpr int kMaxDevices = 64;
    static std::atomic<uint32_t *> addr[kMaxDevices] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    uint32_t *a = addr[dev].load(std::memory_order_acquire);
    if (!a) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_slot_of) != cudaSuccess || !p) return nullptr;
        a = static_cast<uint32_t *>(p);
        addr[dev].store(a, std::memory_order_release);
    }
    return a;
}

}  // namespace

namespace kvgov_host {

// Owner min of a batch whose keys a fused chain kernel has inserted (one
// thread per request; see owner_min_req_kernel).
int arrival_owner_min_by_request(const int64_t *d_blk_off, int32_t n_req, uint32_t *d_slot_of,
                                 uint64_t *d_owner, uint64_t seq_base, cudaStream_t stream) {
    const unsigned grid = (unsigned)(((long long)n_req + kThreads - 1) / kThreads);
    owner_min_req_kernel<<<grid, kThreads, 0, stream>>>(d_blk_off, n_req, d_slot_of,
                                                        reinterpret_cast<unsigned long long *>(d_owner), seq_base);
    return launch_status();
}

bool arrival_args_ok(uint64_t capacity, uint64_t seq_base) {
    return arrival_capacity(capacity) && seq_base != 0 && seq_base <= kMaxSeq;
}

}  // namespace kvgov_host

// The blocks of the batch's first kFirstRequests requests, inserted before
// the rest.  Requests that share a prefix (a system prompt, a template) all
// hold its keys; inserted by every thread at once, each such key would see
// thousands of compare-and-swaps race on one slot.  Inserted first, the keys
// are in the table when the other threads read their slots, and those finish
// with plain reads.  The owners stay exact: these blocks come first in
// arrival order, and the owner min settles any later copy.
// Only batches of kFirstMinBatch requests or more take this pass: with fewer
// requests per shared key the race is short and the extra launch costs more
// than it saves (measured: template batch of 8192 requests, unsalted 46 -> 28
// us; 256 to 1024 requests, 4-8 us slower with the pass).
constexpr int32_t kFirstRequests = 32;
constexpr int32_t kFirstMinBatch = 4096;

static void insert_first_requests(uint8_t *d_slots, uint64_t capacity, uint64_t *d_owner, const uint8_t *d_digests,
                           const int64_t *d_blk_off, int32_t n_req, uint32_t *slot_of, unsigned long long *d_n_new,
                           uint32_t *d_status, long long row_cap, uint64_t seq_base, cudaStream_t s) {
    if (n_req < kFirstMinBatch) return;
    const int32_t first = kFirstRequests;
    insert_arrival_kernel<<<kvgov_host::sm_count(), kThreads, 0, s>>>(
        reinterpret_cast<unsigned long long *>(d_slots), capacity - 1, reinterpret_cast<unsigned long long *>(d_owner),
        reinterpret_cast<const uint4 *>(d_digests), d_blk_off, n_req, slot_of, d_n_new, d_status,
        kvgov_host::spin_limit(), row_cap, seq_base, first);
}

extern "C" int kvgov_owner_init(uint64_t *d_owner, uint64_t capacity, kvgov_stream_t stream) {
    if (!d_owner || !kvgov_host::aligned16(d_owner) || !arrival_capacity(capacity)) return KVGOV_EINVAL;
    const unsigned long long n_vec = (capacity + KVGOV_STASH_SLOTS) / 2;   // main slots and side store: whole uint4s
    const unsigned long long want = (n_vec + 255) / 256;
    const unsigned long long cap = (unsigned long long)kvgov_host::sm_count() * 16;
    const unsigned grid = (unsigned)(want < cap ? want : cap);
    owner_init_kernel<<<grid, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(reinterpret_cast<uint4 *>(d_owner),
                                                                                 n_vec);
    return kvgov_host::launch_status();
}

extern "C" int kvgov_insert_arrival(uint8_t *d_slots, uint64_t *d_owner, uint64_t capacity, const uint8_t *d_digests,
                                    const int64_t *d_blk_off, int32_t n_req, uint64_t seq_base, uint32_t *d_slot_of,
                                    unsigned long long *d_n_new, uint32_t *d_status, kvgov_stream_t stream) {
    using kvgov_host::aligned16;
    if (!d_slots || !aligned16(d_slots) || !d_owner || !arrival_capacity(capacity) || n_req < 0 || !d_status ||
        seq_base == 0 || seq_base > kMaxSeq)
        return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;
    if (!d_digests || !aligned16(d_digests) || !d_blk_off || !d_slot_of) return KVGOV_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const unsigned grid = row_grid();
    insert_first_requests(d_slots, capacity, d_owner, d_digests, d_blk_off, n_req, d_slot_of, d_n_new, d_status,
                          kNoRowCap, seq_base, s);
    insert_arrival_kernel<<<grid, kThreads, 0, s>>>(reinterpret_cast<unsigned long long *>(d_slots), capacity - 1,
                                                    reinterpret_cast<unsigned long long *>(d_owner),
                                                    reinterpret_cast<const uint4 *>(d_digests), d_blk_off, n_req,
                                                    d_slot_of, d_n_new, d_status, kvgov_host::spin_limit(),
                                                    kNoRowCap, seq_base, 0);
    owner_min_kernel<<<grid, kThreads, 0, s>>>(d_blk_off, n_req, d_slot_of,
                                               reinterpret_cast<unsigned long long *>(d_owner), seq_base, kNoRowCap);
    return kvgov_host::launch_status();
}

extern "C" int kvgov_probe_arrival(const uint64_t *d_owner, uint64_t capacity, const uint32_t *d_slot_of,
                                   const int64_t *d_blk_off, int32_t n_req, uint64_t seq_base,
                                   int32_t *d_prefix_blocks, uint32_t *d_status, kvgov_stream_t stream) {
    if (!d_owner || !arrival_capacity(capacity) || n_req < 0 || seq_base == 0 || seq_base > kMaxSeq)
        return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;
    if (!d_slot_of || !d_blk_off || !d_prefix_blocks) return KVGOV_EINVAL;
    probe_arrival_kernel<<<request_grid(n_req), kThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<const unsigned long long *>(d_owner), d_slot_of, d_blk_off, n_req, seq_base,
        d_prefix_blocks, d_status, kNoRowCap);
    return kvgov_host::launch_status();
}

extern "C" int kvgov_serve_arrival_static(uint8_t *d_slots, uint64_t *d_owner, uint64_t capacity,
                                          const uint8_t *d_digests, const int64_t *d_blk_off, int32_t n_req,
                                          int64_t n_blocks, uint64_t seq_base, int32_t *d_prefix_blocks,
                                          unsigned long long *d_n_new, uint32_t *d_status, kvgov_stream_t stream) {
    using kvgov_host::aligned16;
    if (!d_slots || !aligned16(d_slots) || !d_owner || !arrival_capacity(capacity) || n_req < 0 || !d_status ||
        seq_base == 0 || seq_base > kMaxSeq || n_blocks < 0 || n_blocks > kStaticRows)
        return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;
    if (!d_digests || !aligned16(d_digests) || !d_blk_off || !d_prefix_blocks) return KVGOV_EINVAL;
    uint32_t *slot_of = static_slot_of();
    if (!slot_of) return KVGOV_ECUDA;
    // Nothing in the scratch has to start at zero: the insert writes the entry
    // of every block that the owner min and the probe read.  Every kernel
    // takes n_blocks (<= kStaticRows) as its row bound, so a batch whose
    // d_blk_off[n_req] exceeds it reads no digest row past n_blocks and
    // touches no scratch entry past it: nothing is inserted and the probe
    // flags every request.
    const long long row_cap = (long long)n_blocks;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const unsigned grid = row_grid();
    insert_first_requests(d_slots, capacity, d_owner, d_digests, d_blk_off, n_req, slot_of, d_n_new, d_status,
                          row_cap, seq_base, s);
    insert_arrival_kernel<<<grid, kThreads, 0, s>>>(reinterpret_cast<unsigned long long *>(d_slots), capacity - 1,
                                                    reinterpret_cast<unsigned long long *>(d_owner),
                                                    reinterpret_cast<const uint4 *>(d_digests), d_blk_off, n_req,
                                                    slot_of, d_n_new, d_status, kvgov_host::spin_limit(), row_cap,
                                                    seq_base, 0);
    owner_min_kernel<<<grid, kThreads, 0, s>>>(d_blk_off, n_req, slot_of,
                                               reinterpret_cast<unsigned long long *>(d_owner), seq_base, row_cap);
    probe_arrival_kernel<<<request_grid(n_req), kThreads, 0, s>>>(reinterpret_cast<const unsigned long long *>(d_owner),
                                                                  slot_of, d_blk_off, n_req, seq_base,
                                                                  d_prefix_blocks, d_status, row_cap);
    return kvgov_host::launch_status();
}
