// kvgov_chain.cu -- the chained, salted block digests (kvgov_chain_hash,
// kvgov_chain_hash_probe, kvgov_chain_hash_arrival,
// kvgov_chain_hash_insert_prev).
//
// Paper: section 2.1 equation (h_0 = H(tokens_0..B-1), h_j = H(h_{j-1},
// tokens_j)), section 4.1 equation (sigma_p prepended at the root) and
// section 4.2 equation (sigma_p prepended at the divergence block k).
//
// Chain kernel layout.  One thread owns one request's chain: the chain is
// sequential in j (each digest feeds the next message), so parallelism comes
// from the batch.  A CTA of kR threads walks block index j in lockstep; for
// every j each thread stages its own request's 64-byte block into shared
// memory with 16-byte cp.async copies (a block starting at a token offset
// that is not a multiple of 4 spans five aligned 16-byte chunks; a thread's
// chunks sit 80 bytes from its neighbours', so eight 16-byte writes hit 32
// distinct banks), double-buffered so that the copy of block j+1 overlaps
// the hashing of block j.  (The CTA's threads sharing out all its chunks, a
// request's chunks on consecutive threads, cost a division, two shared
// loads and the address arithmetic per chunk: the wide batch's step 0.2243
// -> 0.2193 ms, the probe-heavy batch's chain with the fused probe 430 ->
// 398 us with each thread on its own chunks.)  Each thread then reads its 16
// tokens from shared memory, byte-swaps them into big-endian SHA words and
// runs the 2 (or 3) compressions of its message in registers.
#include "kvgov_insert.cuh"
#include "kvgov_internal.cuh"
#include "kvgov_lookup.cuh"
#include "sha256_dev.cuh"

namespace {

using namespace kvgov_dev;

struct DeviceInfo {
    int sms = 0;
};

// SM count of the current device, looked up once per device.
DeviceInfo device_info() {
    static DeviceInfo cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return DeviceInfo{};
    DeviceInfo &d = cache[dev];
    if (d.sms == 0) {
        int sms = 0;
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        d.sms = sms;
    }
    return d;
}

// ---------------------------------------------------------------------------
// Chain kernel
// ---------------------------------------------------------------------------

constexpr int kR = 128;           // requests (threads) per CTA
constexpr int kStages = 2;        // shared-memory buffers for token blocks
constexpr int kChunks = 5;        // 16-byte chunks that can cover one 64-byte block
constexpr int kSlotWords = kChunks * 4;

struct ChainParams {
    const int32_t *tokens;
    const int64_t *tok_off;
    const int32_t *principal;
    const uint8_t *salts;
    const int32_t *boundary_tok;
    const int64_t *blk_off;
    uint8_t *digests;
    uint32_t *status;
    int32_t n_req;
    int32_t n_principals;
    // fused probe (kvgov_chain_hash_probe) and fused arrival insert
    // (kvgov_chain_hash_arrival) only
    const uint4 *slots;
    unsigned long long mask;
    int32_t *prefix_blocks;
};

// The fused arrival insert's own arguments (a separate kernel parameter, so
// that the other variants keep their parameter block).
struct ArrivalParams {
    unsigned long long *owner = nullptr;
    uint32_t *slot_of = nullptr;
    unsigned long long *n_new = nullptr;
    unsigned long long seq_base = 0;
    uint32_t spin_limit = 0;
};

// The previous batch whose uncached blocks kFuseInsertPrev inserts.
struct PrevParams {
    unsigned long long *slots = nullptr;
    unsigned long long mask = 0;
    const uint4 *digests = nullptr;
    const int64_t *blk_off = nullptr;
    const int32_t *prefix_blocks = nullptr;
    int32_t n_req = 0;
    unsigned long long *n_new = nullptr;
    uint32_t spin_limit = 0;
};

// The generations of kFuseServe: per handle (slot, or capacity + 8 + side-
// store entry) the generation of the batch that claimed it; a key counts as
// cached for this batch iff floor <= its generation < g.
struct GenParams {
    uint32_t *gen = nullptr;
    uint32_t g = 0;
    uint32_t floor = 0;
    unsigned long long *n_new = nullptr;
    uint32_t spin_limit = 0;
};

// What the chain kernel does with each digest besides storing it.
constexpr int kFuseNone = 0;      // nothing (kvgov_chain_hash)
constexpr int kFuseProbe = 1;     // look it up (kvgov_chain_hash_probe)
constexpr int kFuseArrival = 2;   // insert it, arrival order (kvgov_chain_hash_arrival)
constexpr int kFuseInsertPrev = 3;   // insert the previous batch's uncached blocks (kvgov_chain_hash_insert_prev)
constexpr int kFuseInsertPrevProbe = 4;   // both: the insert, and a lookup giving a lower bound of the prefix
constexpr int kFuseServe = 5;        // look it up among older batches' keys, insert it if past the prefix
                                     // (kvgov_chain_hash_serve)

// Big-endian words of principal pi's 32-byte salt.
__device__ __forceinline__ void load_salt(const uint8_t *salts, int pi, uint32_t sw[8]) {
    const uint4 *s = reinterpret_cast<const uint4 *>(salts + 32ll * pi);
    const uint4 a = __ldg(s), b = __ldg(s + 1);
    sw[0] = bswap32(a.x); sw[1] = bswap32(a.y); sw[2] = bswap32(a.z); sw[3] = bswap32(a.w);
    sw[4] = bswap32(b.x); sw[5] = bswap32(b.y); sw[6] = bswap32(b.z); sw[7] = bswap32(b.w);
}

// kFuseProbe: after storing block j's digest, a thread whose blocks 0..j-1
// were all found in the table looks block j up too (kvgov_probe's
// definition), and at the end writes its request's cached-prefix length.
// kFuseArrival: block j's key goes into the table at once (the insert of
// kvgov_insert_arrival): the lanes of a warp hold block j of 32 consecutive
// requests, so a key their prefixes share is inserted by its lowest lane
// only and the others take its slot.  Either way the memory latency is
// covered by the other warps' hashing.
// kFuseInsertPrev: thread t inserts the uncached blocks of the previous
// batch's requests t, t + T, ... (T threads in the grid), one block per
// iteration of its own chain and the rest after it (the insert of
// kvgov_insert_uncached).
// kFuseInsertPrevProbe: the insert of kFuseInsertPrev and the lookups of
// kFuseProbe in one launch.  A lookup that runs while the insert fills the
// table can miss a key that is being inserted (it reads an empty slot or a
// claimed slot whose second half is not yet written) but never finds one
// that is absent, since a slot, once claimed, never changes its key.  So
// the prefix it leaves is a lower bound of the prefix on the table after the
// insert, and a probe that resumes each walk where it stopped
// (kvgov_host::probe_resume) makes it exact.
// kFuseServe: the batch's own lookups and insert in one launch.  A thread
// whose blocks 0..j-1 were all cached looks block j up, and counts it as
// cached only if the generation of the key's slot is in [floor, g): written
// by an earlier batch since the last flush.  From the first block that is
// not cached on, the blocks are inserted -- but for one that the lookup found
// already added by this batch -- and a slot claimed gets generation g, written
// after the claim; the first such block's insert starts its walk where the
// lookup's stopped.  No ordering between the two is needed: a slot that this launch
// claims was empty when the launch began, so its generation then was below
// floor (never written since the flush), and a lookup reads either that or
// g -- both "not cached", as they should be for a key of this batch; and
// keys of earlier launches, with their generations, are all visible.  The
// prefix lengths are those of kvgov_probe before the batch's insert, the
// table and key count those of kvgov_insert_uncached after it.
template <int MODE, int FUSE>
__device__ __forceinline__ void chain_body(const ChainParams &p, const ArrivalParams &a,
                                           const PrevParams &q = PrevParams{}, const GenParams &gp = GenParams{}) {
    __shared__ __align__(16) uint32_t stage[kStages][kR * kSlotWords];
    __shared__ int s_jmax;
    __shared__ unsigned int s_new, s_flags, s_done;   // kFuseArrival counts

    const int tid = threadIdx.x;
    const long long r = (long long)blockIdx.x * kR + tid;
    // The variants that insert keep the CTA in step, block by block: without
    // that barrier the serving step's chain launch took 498 us against 190
    // (a mean over steps that include cache flushes, where every request
    // inserts the same shared-prefix keys) and the arrival-order call 234
    // against 212 us.  The others need none (next comment).
    constexpr bool kIns = FUSE == kFuseInsertPrev || FUSE == kFuseInsertPrevProbe;   // the previous batch's insert
    constexpr bool kLook = FUSE == kFuseProbe || FUSE == kFuseInsertPrevProbe;        // lookups of this batch
    constexpr bool kServe = FUSE == kFuseServe;
    constexpr bool kLockstep = FUSE == kFuseArrival || kIns || kServe;
    if (kLockstep && tid == 0) { s_new = 0; s_flags = 0; s_done = 0; s_jmax = 0; }

    // Per-request set-up and validation.
    const long long tok_end = p.tok_off[p.n_req];
    long long t0 = 0, row = 0;
    int nb = 0, k = -1, pi = 0;
    if (r < p.n_req) {
        t0 = p.tok_off[r];
        const long long t1 = p.tok_off[r + 1];
        const long long nbl = (t1 - t0) / KVGOV_BLOCK;
        bool ok = t0 >= 0 && t1 >= t0 && t1 <= tok_end && nbl < (1ll << 31);
        row = p.blk_off[r];
        ok = ok && row >= 0 && p.blk_off[r + 1] - row == nbl && row + nbl <= p.blk_off[p.n_req];
        if (MODE != KVGOV_UNSALTED) {
            pi = p.principal[r];
            ok = ok && pi >= 0 && pi < p.n_principals;
        }
        if (MODE == KVGOV_ROOT) k = 0;
        if (MODE == KVGOV_BOUNDARY) {
            const int b = p.boundary_tok[r];
            ok = ok && b >= 0;
            k = b / KVGOV_BLOCK;
        }
        if (ok) nb = (int)nbl;
        else raise_flag(p.status, KVGOV_F_BADINDEX);
    }
    // Each thread stages and reads only its own request's blocks, so the
    // warps of a CTA need no barrier between blocks: a warp held up by a
    // fused lookup holds back no other (the probe-heavy batch's chain with
    // the fused probe: 397 -> 380 us), and the lanes of a warp walk the
    // warp's longest chain.  With kLockstep the CTA walks its longest.
    int jmax;
    if (kLockstep) {
        __syncthreads();
        if (nb > 0) atomicMax(&s_jmax, nb);
        __syncthreads();
        jmax = s_jmax;
    } else {
        jmax = (int)__reduce_max_sync(0xffffffffu, (unsigned)nb);
    }

    // Stage this thread's request's block jj into buffer buf.
    const char *tok_bytes = reinterpret_cast<const char *>(p.tokens);
    const long long end_bytes = tok_end * 4;
    auto issue = [&](int jj, int buf) {
        if (jj < nb) {
            const long long sb = (t0 + (long long)KVGOV_BLOCK * jj) * 4;
            const long long a0 = sb & ~15ll;
#pragma unroll
            for (int c = 0; c < kChunks; ++c) {
                if (c == kChunks - 1 && a0 == sb) break;      // aligned block: four chunks
                const long long ca = a0 + 16ll * c;
                const long long avail = end_bytes - ca;
                cp_async16(&stage[buf][tid * kSlotWords + c * 4], tok_bytes + ca, avail >= 16 ? 16 : (int)avail);
            }
        }
    };

#pragma unroll
    for (int s = 0; s < kStages - 1; ++s) {
        if (s < jmax) issue(s, s);
        cp_async_commit();
    }

    // Plain adds: measured on GB300, issuing them as IMAD (AddFma) only adds
    // instructions, since IMAD shares the integer pipe with SHF, LOP3 and
    // IADD3 (libkvgov_peak kinds 3-5).
    const AddAlu add{};
    const int sh = (int)(t0 & 3);   // word offset of the block inside its first chunk
    uint32_t h[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) h[i] = 0u;
    int hits = 0;   // kFuseProbe: leading blocks found in the table so far
    unsigned my_new = 0, my_flags = 0;   // kFuseArrival

    unsigned long long ak[4] = {0ull, 0ull, 0ull, 0ull};   // kFuseArrival: block j's key
    bool have = false;                                      // ... to be inserted by this lane

    // kFuseInsertPrev: the previous batch's request pq this thread inserts,
    // its next uncached row and how many of its uncached blocks remain.
    const long long pstride = (long long)gridDim.x * kR;
    long long pq = r, prow = 0;
    long long pleft = 0;
    auto prev_next = [&]() {                     // from pq on: the first request with uncached blocks
        for (; pq < q.n_req; pq += pstride) {
            const long long base = q.blk_off[pq], pnb = q.blk_off[pq + 1] - base;
            if (pnb < 0 || base < 0 || base + pnb > q.blk_off[q.n_req]) {
                my_flags |= KVGOV_F_BADINDEX;
                continue;
            }
            long long L = q.prefix_blocks[pq];
            L = L < 0 ? 0 : (L > pnb ? pnb : L);
            if (pnb > L) {
                prow = base + L;
                pleft = pnb - L;
                return;
            }
        }
        pleft = 0;
    };
    auto prev_insert_one = [&]() {               // insert row prow of the previous batch
        const uint4 x = __ldg(q.digests + 2 * prow), y = __ldg(q.digests + 2 * prow + 1);
        const unsigned long long key[4] = {u64_of(x.x, x.y), u64_of(x.z, x.w), u64_of(y.x, y.y), u64_of(y.z, y.w)};
        if (key_is_zero(key)) {
            my_flags |= KVGOV_F_SENTINEL;
        } else {
            unsigned long long pos = 0;
            count_insert(insert_one(q.slots, q.mask, key, q.spin_limit, &pos), my_new, my_flags);
        }
        ++prow;
        if (--pleft == 0) {
            pq += pstride;
            prev_next();
        }
    };
    if (kIns) prev_next();
    for (int j = 0; j < jmax; ++j) {
        const int jn = j + kStages - 1;
        if (jn < jmax) issue(jn, jn % kStages);
        cp_async_commit();
        cp_async_wait<kStages - 1>();      // this thread's copies of block j have landed
        if (kLockstep) __syncthreads();

        if (j < nb) {
            const uint32_t *src = &stage[j % kStages][tid * kSlotWords + sh];
            uint32_t tw[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) tw[i] = bswap32(src[i]);

            if (MODE == KVGOV_UNSALTED) {
                if (j == 0) sha256_msg64(tw, h, add);
                else sha256_msg96(h, tw, h, add);
            } else if (MODE == KVGOV_ROOT) {
                uint32_t pw[8];
                if (j == 0) load_salt(p.salts, pi, pw);
                else {
#pragma unroll
                    for (int i = 0; i < 8; ++i) pw[i] = h[i];
                }
                sha256_msg96(pw, tw, h, add);
            } else {
                if (j == k && j > 0) {
                    uint32_t sw[8];
                    load_salt(p.salts, pi, sw);
                    sha256_msg128(sw, h, tw, h, add);
                } else if (j == 0 && k != 0) {
                    sha256_msg64(tw, h, add);
                } else {
                    uint32_t pw[8];
                    if (j == k) load_salt(p.salts, pi, pw);
                    else {
#pragma unroll
                        for (int i = 0; i < 8; ++i) pw[i] = h[i];
                    }
                    sha256_msg96(pw, tw, h, add);
                }
            }

            uint4 *dst = reinterpret_cast<uint4 *>(p.digests + (row + j) * 32);
            const uint4 q0 = make_uint4(bswap32(h[0]), bswap32(h[1]), bswap32(h[2]), bswap32(h[3]));
            const uint4 q1 = make_uint4(bswap32(h[4]), bswap32(h[5]), bswap32(h[6]), bswap32(h[7]));
            dst[0] = q0;
            dst[1] = q1;
            if (kLook && hits == j && lookup(p.slots, p.mask, q0, q1)) hits = j + 1;
            if (kServe) {
                // -1 not looked up or not found, 0 found but added by this batch, 1 cached
                int found = -1;
                unsigned long long start = 0;            // where the insert's walk may begin
                if (hits == j) found = lookup_serve(p.slots, p.mask, gp.gen, gp.floor, gp.g, q0, q1, &start);
                if (found == 1) {
                    hits = j + 1;
                } else if (found < 0) {                  // past the prefix and not in the table yet: insert
                    const unsigned long long key[4] = {u64_of(q0.x, q0.y), u64_of(q0.z, q0.w), u64_of(q1.x, q1.y),
                                                       u64_of(q1.z, q1.w)};
                    if (key_is_zero(key)) {
                        my_flags |= KVGOV_F_SENTINEL;
                    } else {
                        unsigned long long pos = 0;
                        const InsertResult res = insert_one(
                            reinterpret_cast<unsigned long long *>(const_cast<uint4 *>(p.slots)), p.mask, key,
                            gp.spin_limit, &pos, start);
                        count_insert(res, my_new, my_flags);
                        if (res == kNew) gp.gen[pos] = gp.g;
                    }
                }
            }
            if (FUSE == kFuseArrival) {
                ak[0] = u64_of(q0.x, q0.y); ak[1] = u64_of(q0.z, q0.w);
                ak[2] = u64_of(q1.x, q1.y); ak[3] = u64_of(q1.z, q1.w);
                have = !key_is_zero(ak);
                if (!have) {
                    my_flags |= KVGOV_F_SENTINEL;
                    a.slot_of[row + j] = kNoSlot;
                }
            }
        }
        if (FUSE == kFuseArrival) {                     // every lane of the warp is here
            const unsigned inserting = __ballot_sync(0xffffffffu, have);
            if (have) {
                const unsigned same = __match_any_sync(inserting, ak[0]) & __match_any_sync(inserting, ak[1]) &
                                      __match_any_sync(inserting, ak[2]) & __match_any_sync(inserting, ak[3]);
                const int leader = __ffs(same) - 1;
                unsigned long long pos = 0ull;
                int res = kDuplicate;
                const bool lead = (tid & 31) == leader;
                if (lead) {
                    res = insert_one(reinterpret_cast<unsigned long long *>(const_cast<uint4 *>(p.slots)), p.mask,
                                     ak, a.spin_limit, &pos);
                    count_insert(static_cast<InsertResult>(res), my_new, my_flags);
                    if (res == kNew) a.owner[pos] = a.seq_base + (unsigned long long)(row + j);
                }
                pos = __shfl_sync(inserting, pos, leader);
                res = __shfl_sync(inserting, res, leader);
                // settled (no owner min needed): the block that claimed the slot,
                // and every block behind an earlier lane with the same key
                const uint32_t mark = (res == kNew || !lead) ? kSettled : 0u;
                a.slot_of[row + j] = (res == kNew || res == kDuplicate) ? ((uint32_t)pos | mark) : kNoSlot;
            }
            have = false;
        }
        if (kIns && pleft > 0) prev_insert_one();
        if (kLockstep) __syncthreads();
    }
    cp_async_wait<0>();
    if ((kLook || kServe) && r < p.n_req) p.prefix_blocks[r] = hits;
    if (kIns)
        while (pleft > 0) prev_insert_one();
    if (FUSE == kFuseArrival || kIns || kServe)
        publish_counts(my_new, my_flags, &s_new, &s_flags, &s_done,
                       FUSE == kFuseArrival ? a.n_new : (kServe ? gp.n_new : q.n_new), p.status);
}

template <int MODE, int FUSE>
__global__ void __launch_bounds__(kR) chain_kernel(const ChainParams p) {
    chain_body<MODE, FUSE>(p, ArrivalParams{});
}

template <int MODE>
__global__ void __launch_bounds__(kR) chain_arrival_kernel(const ChainParams p, const ArrivalParams a) {
    chain_body<MODE, kFuseArrival>(p, a);
}

// At most 64 registers, so that 8 CTAs fit an SM: the batch's CTAs leave
// room beside them for the next batch's salts and block offsets.
// FUSE: kFuseInsertPrev or kFuseInsertPrevProbe.
template <int MODE, int FUSE>
__global__ void __launch_bounds__(kR, 8) chain_prev_kernel(const ChainParams p, const PrevParams q) {
    chain_body<MODE, FUSE>(p, ArrivalParams{}, q);
}

// kFuseServe; at most 64 registers, as chain_prev_kernel.
template <int MODE>
__global__ void __launch_bounds__(kR, 8) chain_serve_kernel(const ChainParams p, const GenParams gp) {
    chain_body<MODE, kFuseServe>(p, ArrivalParams{}, PrevParams{}, gp);
}

}  // namespace

namespace {

// Launch chain_kernel<mode, FUSE> (chain_arrival_kernel<mode> for kFuseArrival,
// chain_prev_kernel<mode, FUSE> for kFuseInsertPrev and kFuseInsertPrevProbe).
template <int FUSE>
void launch_chain_kernel(int mode, unsigned grid, cudaStream_t s, const ChainParams &p,
                         const ArrivalParams &a = ArrivalParams{}, const PrevParams &q = PrevParams{}) {
    if constexpr (FUSE == kFuseInsertPrev || FUSE == kFuseInsertPrevProbe) {
        switch (mode) {
        case KVGOV_UNSALTED: chain_prev_kernel<KVGOV_UNSALTED, FUSE><<<grid, kR, 0, s>>>(p, q); break;
        case KVGOV_ROOT: chain_prev_kernel<KVGOV_ROOT, FUSE><<<grid, kR, 0, s>>>(p, q); break;
        default: chain_prev_kernel<KVGOV_BOUNDARY, FUSE><<<grid, kR, 0, s>>>(p, q); break;
        }
    } else if constexpr (FUSE == kFuseArrival) {
        switch (mode) {
        case KVGOV_UNSALTED: chain_arrival_kernel<KVGOV_UNSALTED><<<grid, kR, 0, s>>>(p, a); break;
        case KVGOV_ROOT: chain_arrival_kernel<KVGOV_ROOT><<<grid, kR, 0, s>>>(p, a); break;
        default: chain_arrival_kernel<KVGOV_BOUNDARY><<<grid, kR, 0, s>>>(p, a); break;
        }
    } else {
        switch (mode) {
        case KVGOV_UNSALTED: chain_kernel<KVGOV_UNSALTED, FUSE><<<grid, kR, 0, s>>>(p); break;
        case KVGOV_ROOT: chain_kernel<KVGOV_ROOT, FUSE><<<grid, kR, 0, s>>>(p); break;
        default: chain_kernel<KVGOV_BOUNDARY, FUSE><<<grid, kR, 0, s>>>(p); break;
        }
    }
}

// The chain hash alone: kvgov_chain_split.cu's kernel for a batch too small
// to fill the GPU (each chain's rounds and schedule on two warps), the
// chain kernel above otherwise.
int launch_plain(int mode, unsigned grid, cudaStream_t s, const ChainParams &p) {
    if (p.n_req <= kvgov_host::chain_split_max_req())
        return kvgov_host::launch_chain_split(mode, p.tokens, p.tok_off, p.n_req, p.principal, p.salts,
                                              p.n_principals, p.boundary_tok, p.blk_off, p.digests, p.status, s);
    launch_chain_kernel<kFuseNone>(mode, grid, s, p);
    return kvgov_host::launch_status();
}

// The table and arrival arguments of the fused variants.
struct FuseArgs {
    int fuse = kFuseNone;
    const uint8_t *slots = nullptr;
    uint64_t capacity = 0;
    int32_t *prefix_blocks = nullptr;   // kFuseProbe
    uint64_t *owner = nullptr;          // kFuseArrival
    uint64_t seq_base = 0;
    uint32_t *slot_of = nullptr;
    unsigned long long *n_new = nullptr;
    const uint8_t *prev_digests = nullptr;     // kFuseInsertPrev
    const int64_t *prev_blk_off = nullptr;
    int32_t prev_n_req = 0;
    const int32_t *prev_prefix_blocks = nullptr;
    int32_t *probe_prefix_blocks = nullptr;     // kFuseInsertPrev: probe this batch after the insert ...
    bool probe_complete = true;                 // ... to the end (else: leave a lower bound, see launch_chain)
    uint32_t *gen = nullptr;                    // kFuseServe: the table's generations, this batch's, the floor
    uint32_t g = 0;
    uint32_t gen_floor = 0;
};

int launch_chain(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                 const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                 const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests, uint32_t *d_status,
                 const FuseArgs &f, kvgov_stream_t stream) {
    using kvgov_host::aligned16;
    if (mode != KVGOV_UNSALTED && mode != KVGOV_ROOT && mode != KVGOV_BOUNDARY) return KVGOV_EINVAL;
    if (n_req < 0) return KVGOV_EINVAL;
    if (!d_tokens || !aligned16(d_tokens) || !d_tok_off || !d_blk_off || !d_digests || !aligned16(d_digests))
        return KVGOV_EINVAL;
    // the per-request arrays are needed only when there are requests
    if (mode != KVGOV_UNSALTED && n_req > 0 &&
        (!d_principal || !d_salts || !aligned16(d_salts) || n_principals <= 0))
        return KVGOV_EINVAL;
    if (mode == KVGOV_BOUNDARY && n_req > 0 && !d_boundary_tok) return KVGOV_EINVAL;
    if (f.fuse == kFuseProbe &&
        (!f.prefix_blocks || !f.slots || !aligned16(f.slots) || !kvgov_host::pow2_capacity(f.capacity)))
        return KVGOV_EINVAL;
    if (f.fuse == kFuseArrival &&
        (!f.prefix_blocks || !f.slots || !aligned16(f.slots) || !f.owner || !f.slot_of || !d_status ||
         !kvgov_host::arrival_args_ok(f.capacity, f.seq_base)))
        return KVGOV_EINVAL;
    if (f.fuse == kFuseInsertPrev &&
        (!f.slots || !aligned16(f.slots) || !kvgov_host::pow2_capacity(f.capacity) || !d_status ||
         f.prev_n_req < 0 ||
         (f.prev_n_req > 0 && (!f.prev_digests || !aligned16(f.prev_digests) || !f.prev_blk_off ||
                               !f.prev_prefix_blocks))))
        return KVGOV_EINVAL;
    // the previous batch's insert alone when this batch is empty
    auto insert_prev = [&]() {
        return kvgov_insert_uncached(const_cast<uint8_t *>(f.slots), f.capacity, f.prev_digests, f.prev_blk_off,
                                     f.prev_n_req, f.prev_prefix_blocks, f.n_new, d_status, stream);
    };
    if (f.fuse == kFuseServe && (!f.slots || !aligned16(f.slots) || !kvgov_host::pow2_capacity(f.capacity) ||
                                 !f.gen || !d_status || (n_req > 0 && !f.prefix_blocks) || f.gen_floor > f.g))
        return KVGOV_EINVAL;
    if (n_req == 0) return (f.fuse == kFuseInsertPrev && f.prev_n_req > 0) ? insert_prev() : KVGOV_OK;

    ChainParams p;
    p.tokens = d_tokens; p.tok_off = d_tok_off; p.principal = d_principal; p.salts = d_salts;
    p.boundary_tok = d_boundary_tok; p.blk_off = d_blk_off; p.digests = d_digests; p.status = d_status;
    p.n_req = n_req; p.n_principals = n_principals;
    p.slots = reinterpret_cast<const uint4 *>(f.slots);
    p.mask = f.fuse != kFuseNone ? f.capacity - 1 : 0;
    p.prefix_blocks = f.prefix_blocks;
    ArrivalParams a;
    a.owner = reinterpret_cast<unsigned long long *>(f.owner);
    a.slot_of = f.slot_of;
    a.n_new = f.n_new;
    a.seq_base = f.seq_base;
    a.spin_limit = kvgov_host::spin_limit();
    PrevParams q;
    q.slots = reinterpret_cast<unsigned long long *>(const_cast<uint8_t *>(f.slots));
    q.mask = p.mask;
    q.digests = reinterpret_cast<const uint4 *>(f.prev_digests);
    q.blk_off = f.prev_blk_off;
    q.prefix_blocks = f.prev_prefix_blocks;
    q.n_req = f.prev_n_req;
    q.n_new = f.n_new;
    q.spin_limit = a.spin_limit;
    const unsigned grid = (unsigned)(((long long)n_req + kR - 1) / kR);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    // A batch too small to give every SM sub-partition two warps leaves each
    // warp alone on its scheduler, where a fused lookup or insert would stall
    // the chain; there they run as separate launches (same results).
    const DeviceInfo dev = device_info();
    const long long min_fused = 2ll * 32 * 4 * (dev.sms > 0 ? dev.sms : 152);
    // kFuseInsertPrev with probe_prefix_blocks: the chain launch looks every
    // block up as it goes (a lower bound, kFuseInsertPrevProbe) and a probe
    // resumes the walks from there; probe_complete = false leaves that probe
    // to the caller (kvgov_host::probe_resume), with 0 as the bound where the
    // launch made no lookups.
    if (f.fuse == kFuseServe) {
        if (n_req >= min_fused) {
            GenParams gp;
            gp.gen = f.gen;
            gp.g = f.g;
            gp.floor = f.gen_floor;
            gp.n_new = f.n_new;
            gp.spin_limit = kvgov_host::spin_limit();
            switch (mode) {
            case KVGOV_UNSALTED: chain_serve_kernel<KVGOV_UNSALTED><<<grid, kR, 0, s>>>(p, gp); break;
            case KVGOV_ROOT: chain_serve_kernel<KVGOV_ROOT><<<grid, kR, 0, s>>>(p, gp); break;
            default: chain_serve_kernel<KVGOV_BOUNDARY><<<grid, kR, 0, s>>>(p, gp); break;
            }
            return kvgov_host::launch_status();
        }
        // a small batch: the chain, the probe (every key in the table is of an
        // older batch), then the insert with this batch's generation
        int rc = launch_plain(mode, grid, s, p);
        if (rc == KVGOV_OK)
            rc = kvgov_probe(f.slots, f.capacity, d_digests, d_blk_off, n_req, f.prefix_blocks, d_status, stream);
        if (rc == KVGOV_OK)
            rc = kvgov_host::insert_uncached_gen(const_cast<uint8_t *>(f.slots), f.capacity, d_digests, d_blk_off,
                                                 n_req, f.prefix_blocks, f.n_new, d_status, f.gen, f.g, stream);
        return rc;
    }
    if (f.fuse == kFuseInsertPrev) {
        int rc;
        bool lower = false;                        // probe_prefix_blocks holds the lookups' lower bound
        if (f.prev_n_req > 0 && n_req >= min_fused) {
            if (f.probe_prefix_blocks) {
                p.prefix_blocks = f.probe_prefix_blocks;
                launch_chain_kernel<kFuseInsertPrevProbe>(mode, grid, s, p, a, q);
                lower = true;
            } else {
                launch_chain_kernel<kFuseInsertPrev>(mode, grid, s, p, a, q);
            }
            rc = kvgov_host::launch_status();
        } else {                                   // a small batch (or no insert): separate launches
            rc = launch_plain(mode, grid, s, p);
            if (rc == KVGOV_OK && f.prev_n_req > 0) rc = insert_prev();
        }
        if (rc != KVGOV_OK || !f.probe_prefix_blocks) return rc;
        if (f.probe_complete)
            return lower ? kvgov_host::probe_resume(f.slots, f.capacity, d_digests, d_blk_off, n_req,
                                                    f.probe_prefix_blocks, d_status, stream)
                         : kvgov_probe(f.slots, f.capacity, d_digests, d_blk_off, n_req, f.probe_prefix_blocks,
                                       d_status, stream);
        if (!lower && cudaMemsetAsync(f.probe_prefix_blocks, 0, sizeof(int32_t) * (size_t)n_req, s) != cudaSuccess)
            return KVGOV_ECUDA;
        return KVGOV_OK;
    }
    const bool none = f.fuse == kFuseNone;
    const bool fused = !none && n_req >= min_fused;
    if (!fused) {
        int rc = launch_plain(mode, grid, s, p);
        if (rc != KVGOV_OK || none) return rc;
        if (f.fuse == kFuseProbe)
            return kvgov_probe(f.slots, f.capacity, d_digests, d_blk_off, n_req, f.prefix_blocks, d_status, stream);
        rc = kvgov_insert_arrival(const_cast<uint8_t *>(f.slots), f.owner, f.capacity, d_digests, d_blk_off, n_req,
                                  f.seq_base, f.slot_of, f.n_new, d_status, stream);
        if (rc != KVGOV_OK) return rc;
        return kvgov_probe_arrival(f.owner, f.capacity, f.slot_of, d_blk_off, n_req, f.seq_base, f.prefix_blocks,
                                   d_status, stream);
    }
    if (f.fuse == kFuseProbe) {
        launch_chain_kernel<kFuseProbe>(mode, grid, s, p);
        return kvgov_host::launch_status();
    }
    launch_chain_kernel<kFuseArrival>(mode, grid, s, p, a);
    int rc = kvgov_host::launch_status();
    if (rc != KVGOV_OK) return rc;
    rc = kvgov_host::arrival_owner_min_by_request(d_blk_off, n_req, f.slot_of, f.owner, f.seq_base, s);
    if (rc != KVGOV_OK) return rc;
    return kvgov_probe_arrival(f.owner, f.capacity, f.slot_of, d_blk_off, n_req, f.seq_base, f.prefix_blocks,
                               d_status, stream);
}

}  // namespace

extern "C" int kvgov_chain_hash(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                                const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                                uint32_t *d_status, kvgov_stream_t stream) {
    return launch_chain(mode, d_tokens, d_tok_off, n_req, d_principal, d_salts, n_principals, d_boundary_tok,
                        d_blk_off, d_digests, d_status, FuseArgs{}, stream);
}

extern "C" int kvgov_chain_hash_probe(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                      const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                                      const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                                      const uint8_t *d_slots, uint64_t capacity, int32_t *d_prefix_blocks,
                                      uint32_t *d_status, kvgov_stream_t stream) {
    FuseArgs f;
    f.fuse = kFuseProbe;
    f.slots = d_slots;
    f.capacity = capacity;
    f.prefix_blocks = d_prefix_blocks;
    return launch_chain(mode, d_tokens, d_tok_off, n_req, d_principal, d_salts, n_principals, d_boundary_tok,
                        d_blk_off, d_digests, d_status, f, stream);
}

extern "C" int kvgov_chain_hash_arrival(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                        const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                                        const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                                        uint8_t *d_slots, uint64_t *d_owner, uint64_t capacity, uint64_t seq_base,
                                        uint32_t *d_slot_of, int32_t *d_prefix_blocks, unsigned long long *d_n_new,
                                        uint32_t *d_status, kvgov_stream_t stream) {
    FuseArgs f;
    f.fuse = kFuseArrival;
    f.slots = d_slots;
    f.capacity = capacity;
    f.prefix_blocks = d_prefix_blocks;
    f.owner = d_owner;
    f.seq_base = seq_base;
    f.slot_of = d_slot_of;
    f.n_new = d_n_new;
    return launch_chain(mode, d_tokens, d_tok_off, n_req, d_principal, d_salts, n_principals, d_boundary_tok,
                        d_blk_off, d_digests, d_status, f, stream);
}

namespace {

FuseArgs insert_prev_args(uint8_t *d_slots, uint64_t capacity, const uint8_t *d_prev_digests,
                          const int64_t *d_prev_blk_off, int32_t prev_n_req, const int32_t *d_prev_prefix_blocks,
                          int32_t *d_prefix_blocks, unsigned long long *d_n_new, bool probe_complete) {
    FuseArgs f;
    f.fuse = kFuseInsertPrev;
    f.probe_prefix_blocks = d_prefix_blocks;
    f.probe_complete = probe_complete;
    f.slots = d_slots;
    f.capacity = capacity;
    f.n_new = d_n_new;
    f.prev_digests = d_prev_digests;
    f.prev_blk_off = d_prev_blk_off;
    f.prev_n_req = prev_n_req;
    f.prev_prefix_blocks = d_prev_prefix_blocks;
    return f;
}

}  // namespace

extern "C" int kvgov_chain_hash_insert_prev(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                            const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                                            const int32_t *d_boundary_tok, const int64_t *d_blk_off,
                                            uint8_t *d_digests, uint8_t *d_slots, uint64_t capacity,
                                            const uint8_t *d_prev_digests, const int64_t *d_prev_blk_off,
                                            int32_t prev_n_req, const int32_t *d_prev_prefix_blocks,
                                            int32_t *d_prefix_blocks, unsigned long long *d_n_new,
                                            uint32_t *d_status, kvgov_stream_t stream) {
    return launch_chain(mode, d_tokens, d_tok_off, n_req, d_principal, d_salts, n_principals, d_boundary_tok,
                        d_blk_off, d_digests, d_status,
                        insert_prev_args(d_slots, capacity, d_prev_digests, d_prev_blk_off, prev_n_req,
                                         d_prev_prefix_blocks, d_prefix_blocks, d_n_new, true),
                        stream);
}

namespace kvgov_host {
int chain_insert_prev_lower(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                            const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                            const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                            uint8_t *d_slots, uint64_t capacity, const uint8_t *d_prev_digests,
                            const int64_t *d_prev_blk_off, int32_t prev_n_req, const int32_t *d_prev_prefix_blocks,
                            int32_t *d_prefix_lower, unsigned long long *d_n_new, uint32_t *d_status,
                            kvgov_stream_t stream) {
    if (!d_prefix_lower && n_req > 0) return KVGOV_EINVAL;
    return launch_chain(mode, d_tokens, d_tok_off, n_req, d_principal, d_salts, n_principals, d_boundary_tok,
                        d_blk_off, d_digests, d_status,
                        insert_prev_args(d_slots, capacity, d_prev_digests, d_prev_blk_off, prev_n_req,
                                         d_prev_prefix_blocks, d_prefix_lower, d_n_new, false),
                        stream);
}
}  // namespace kvgov_host

extern "C" int kvgov_chain_hash_serve(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                      const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                                      const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                                      uint8_t *d_slots, uint64_t capacity, uint32_t *d_gen, uint32_t gen,
                                      uint32_t gen_floor, int32_t *d_prefix_blocks, unsigned long long *d_n_new,
                                      uint32_t *d_status, kvgov_stream_t stream) {
    FuseArgs f;
    f.fuse = kFuseServe;
    f.slots = d_slots;
    f.capacity = capacity;
    f.prefix_blocks = d_prefix_blocks;
    f.n_new = d_n_new;
    f.gen = d_gen;
    f.g = gen;
    f.gen_floor = gen_floor;
    return launch_chain(mode, d_tokens, d_tok_off, n_req, d_principal, d_salts, n_principals, d_boundary_tok,
                        d_blk_off, d_digests, d_status, f, stream);
}
