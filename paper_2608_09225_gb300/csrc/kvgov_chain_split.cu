// kvgov_chain_split.cu -- the chain hash of a batch too small to fill the
// GPU (the chain launch of kvgov_chain_hash and of its fused variants when
// the batch has at most kvgov_host::chain_split_max_req() requests).
//
// Paper: section 2.1 equation (h_0 = H(tokens_0..B-1), h_j = H(h_{j-1},
// tokens_j)), section 4.1 equation (sigma_p prepended at the root) and
// section 4.2 equation (sigma_p prepended at the divergence block k); the
// digests are the ones kvgov_chain.cu computes.
//
// Why a second kernel.  A chain is sequential in its blocks, so parallelism
// comes only from the batch.  A batch of a few thousand requests gives each
// SM sub-partition one warp (or none), and a warp alone there runs at the
// pace of its own instruction stream: at best one integer instruction every
// two cycles (the integer pipe is 16 lanes wide), in practice slower, since
// each instruction waits on the one it depends on (measured: a lone warp
// takes 35 cycles per SHA-256 round with K_t + W_t in registers, two warps
// sharing a sub-partition 27 each).  Its time per block then grows with the
// instructions on its path, about 2900 for the two compressions with their
// message schedules.  Here the work of 32 chains is split over two warps on
// two sub-partitions:
//   * the round warp runs only the 64 rounds of each compression (about 14
//     integer instructions a round) with K_t + W_t read from shared memory;
//   * the schedule warp stages the tokens (cp.async, two blocks ahead),
//     builds each compression's message (tokens, salt, the previous digest
//     or padding), expands its schedule into K_t + W_t in shared memory, and
//     stores the digests.
// The round warp's work per block drops to about 1800 integer instructions;
// the schedule warp's (about 1300) runs beside it.
//
// Hand-off per block j, on named barriers of 64 threads (one warp arrives,
// the other waits):
//   E0, E1  schedule -> round (E_{j mod 2}, waited on at the start of block
//           j): K_t + W_t of block j's whole second compression, whose
//           message holds no digest, and of the first 16 rounds of its first
//           compression with every word that is h_{j-1} left out -- the round
//           warp adds h_{j-1} itself, so block j starts without waiting for
//           the schedule warp.  Built one block ahead into the other buffer.
//   H       round -> schedule: h_j is in shared memory;
//   B..D    schedule -> round: K_t + W_t of block j's first compression for
//           t in [16q, 16q + 16), chunk q = 1..3 (from h_{j-1} on, so the
//           schedule warp starts them after H).
// Both warps of a pair run the same number of blocks (the pair's longest
// chain) and execute each barrier once per block, so every wait is matched
// by exactly one arrival; a buffer is rewritten only after the wait that
// proves the round warp is done with it.
#include "kvgov_internal.cuh"
#include "kvgov_split.cuh"
#include "sha256_dev.cuh"

namespace {

using namespace kvgov_dev;

constexpr int kPairs = 2;                   // round/schedule warp pairs per CTA
constexpr int kThreads = 64 * kPairs;
constexpr int kChainsPerCta = 32 * kPairs;
constexpr int kTokStages = 3;               // token buffers: blocks j, j + 1 and j + 2 in flight
constexpr int kChunks = 5;                  // 16-byte chunks that cover one 64-byte block

// Shared memory of one pair.  K_t + W_t is stored as uint4 [t / 4][lane], so
// that the round warp reads four rounds' values with one 16-byte load.
struct PairSmem {
    uint4 kw1[12][32];              // first compression of the current block, t = 16..63
    uint4 pm[2][4][32];             // its t = 0..15 without h_{j-1}, by block parity
    uint4 kw2[2][16][32];           // second compression, by block parity
    uint4 h[2][32];                 // the round warp's state after the block
    uint4 tok[kTokStages][32][kChunks];
};
constexpr size_t kSmemBytes = sizeof(PairSmem) * kPairs;

struct SplitParams {
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
};

// What block j's message is, per section 2.1 / 4.1 / 4.2.
constexpr int kSteadyH = 0;      // H(h_{j-1} || T_j)
constexpr int kSteadySalt = 1;   // H(sigma_p || T_0)
constexpr int kFirst = 2;        // H(T_0), unsalted root
constexpr int kBoundary = 3;     // H(sigma_p || h_{k-1} || T_k), k >= 1

template <int MODE>
__device__ __forceinline__ int block_kind(int j, int k) {
    if (MODE == KVGOV_UNSALTED) return j == 0 ? kFirst : kSteadyH;
    if (MODE == KVGOV_ROOT) return j == 0 ? kSteadySalt : kSteadyH;
    if (j == 0) return k == 0 ? kSteadySalt : kFirst;
    return j == k ? kBoundary : kSteadyH;
}

// K_t + W_t of the padding block that ends a 128-byte message (the boundary
// block's third compression): FIPS 180-4 section 5.1.1 padding (0x80, zeros,
// the 64-bit bit length 1024) and section 6.2.2 step 1, evaluated by the
// compiler.
struct PadSchedule {
    uint32_t kw[64];
};
constexpr uint32_t rotr_c(uint32_t x, int n) { return (x >> n) | (x << (32 - n)); }
constexpr PadSchedule pad_schedule(uint32_t bytes) {
    PadSchedule r{};
    uint32_t w[64] = {};
    w[0] = 0x80000000u;
    w[15] = bytes * 8u;
    for (int t = 16; t < 64; ++t) {
        const uint32_t s0 = rotr_c(w[t - 15], 7) ^ rotr_c(w[t - 15], 18) ^ (w[t - 15] >> 3);
        const uint32_t s1 = rotr_c(w[t - 2], 17) ^ rotr_c(w[t - 2], 19) ^ (w[t - 2] >> 10);
        w[t] = w[t - 16] + s0 + w[t - 7] + s1;
    }
    for (int t = 0; t < 64; ++t) r.kw[t] = kShaKHost[t] + w[t];
    return r;
}
__constant__ PadSchedule c_pad128 = pad_schedule(128);

// The round warp's 16 rounds (sha256_dev.cuh).  Another grouping of the
// sums (sha_rounds16_short) measured the same on a lone warp (libkvgov_peak
// kinds 6, 7).
__device__ __forceinline__ void rounds16(uint32_t v[8], const uint32_t kw[16]) { sha_rounds16_t1t2(v, kw); }

// The boundary block's third compression, the constant padding block, out
// of the round warp's loop: a chain runs it once, and kept inline its code
// sat inside the loop every other block runs.
struct State8 {
    uint32_t w[8];
};
static __device__ __noinline__ State8 padding_compression(State8 s) {
    uint32_t v[8], kw[16];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = s.w[i];
#pragma unroll 1
    for (int q = 0; q < 4; ++q) {
#pragma unroll
        for (int i = 0; i < 16; ++i) kw[i] = c_pad128.kw[16 * q + i];
        rounds16(v, kw);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) s.w[i] += v[i];
    return s;
}

// The first chunk of a steady block's first-compression schedule (W_16 ..
// W_31) is what the round warp waits for after its first 16 rounds, and
// half its words are h_{j-1}, known only then.  The terms the tokens
// (words 8..15) fix alone are summed before: W_16 and W_17's
// sigma1(W_14 / W_15) + W_9 / W_10, W_23's sigma0(W_8), and W_t + sigma0(W_{t+1})
// of W_24 .. W_30; the same sums in another order (mod 2^32), the same words.
struct SteadyPre {
    uint32_t t0, t1, t7, t8[7];
};
__device__ __forceinline__ void steady_pre(const uint32_t w[16], SteadyPre &p) {
    p.t0 = ssig1(w[14]) + w[9];
    p.t1 = ssig1(w[15]) + w[10];
    p.t7 = ssig0(w[8]);
#pragma unroll
    for (int i = 0; i < 7; ++i) p.t8[i] = w[8 + i] + ssig0(w[9 + i]);
}
// w: the message (h_{j-1} in words 0..7) -> W_16 .. W_31, as schedule_chunk.
__device__ __forceinline__ void steady_chunk1(uint32_t w[16], const SteadyPre &p) {
    w[0] = w[0] + ssig0(w[1]) + p.t0;
    w[1] = w[1] + ssig0(w[2]) + p.t1;
#pragma unroll
    for (int t = 2; t < 7; ++t) w[t] = w[t] + ssig0(w[t + 1]) + w[t + 9] + ssig1(w[t - 2]);
    w[7] = w[7] + p.t7 + w[0] + ssig1(w[5]);
#pragma unroll
    for (int t = 8; t < 15; ++t) w[t] = p.t8[t - 8] + w[t - 7] + ssig1(w[t - 2]);
    w[15] = w[15] + ssig0(w[0]) + w[8] + ssig1(w[13]);
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1) chain_split_kernel(const SplitParams p) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int pair = warp >> 1;
    const bool round_warp = (warp & 1) == 0;
    PairSmem &sm = reinterpret_cast<PairSmem *>(smem_raw)[pair];
    const int bar_h = 1 + 6 * pair, bar_b = bar_h + 1, bar_e = bar_h + 4;   // B..D = bar_b + 0..2, E0/E1 = bar_e + 0/1

    // Per-chain set-up (both warps of the pair hold the same chain in the same lane).
    const long long r = (long long)blockIdx.x * kChainsPerCta + pair * 32 + lane;
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
        else if (!round_warp) raise_flag(p.status, KVGOV_F_BADINDEX);
    }
    const int jmax = (int)__reduce_max_sync(0xffffffffu, (unsigned)nb);   // the same in both warps

    if (round_warp) {
        uint32_t hp[8];   // h_{j-1}
#pragma unroll
        for (int i = 0; i < 8; ++i) hp[i] = 0u;
        for (int j = 0; j < jmax; ++j) {
            bar_sync(bar_e + (j & 1));
            uint32_t s[8], v[8], kw[16];
            load16(sm.pm[j & 1], lane, kw);
            const int kind = block_kind<MODE>(j, k);
            if (kind == kSteadyH) {            // h_{j-1} is message words 0..7
#pragma unroll
                for (int i = 0; i < 8; ++i) kw[i] += hp[i];
            } else if (kind == kBoundary) {    // words 8..15, after the salt
#pragma unroll
                for (int i = 0; i < 8; ++i) kw[8 + i] += hp[i];
            }
            sha_iv(s);
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] = s[i];
            rounds16(v, kw);
#pragma unroll 1
            for (int q = 1; q < 4; ++q) {
                bar_sync(bar_b + q - 1);
                load16(sm.kw1 + 4 * (q - 1), lane, kw);
                rounds16(v, kw);
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) { s[i] += v[i]; v[i] = s[i]; }
            // second compression: the whole schedule is there since E, so each
            // chunk's values are loaded while the previous chunk's rounds run
            // (two register sets, no copies)
            const uint4 (*k2)[32] = sm.kw2[j & 1];
            uint32_t kb[16];
            load16(k2, lane, kw);
#pragma unroll 1
            for (int q = 0; q < 4; q += 2) {
                load16(k2 + 4 * (q + 1), lane, kb);
                rounds16(v, kw);
                if (q + 2 < 4) load16(k2 + 4 * (q + 2), lane, kw);
                rounds16(v, kb);
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) s[i] += v[i];
            // the boundary block's padding block
            if (MODE == KVGOV_BOUNDARY && __any_sync(0xffffffffu, j > 0 && j == k && j < nb)) {
                State8 st;
#pragma unroll
                for (int i = 0; i < 8; ++i) st.w[i] = s[i];
                st = padding_compression(st);
                if (j > 0 && j == k && j < nb) {
#pragma unroll
                    for (int i = 0; i < 8; ++i) s[i] = st.w[i];
                }
            }
            sm.h[0][lane] = make_uint4(s[0], s[1], s[2], s[3]);
            sm.h[1][lane] = make_uint4(s[4], s[5], s[6], s[7]);
            bar_arrive(bar_h);
#pragma unroll
            for (int i = 0; i < 8; ++i) hp[i] = s[i];
        }
        return;
    }

    // Schedule warp.
    uint32_t sw[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) sw[i] = 0u;
    if (MODE != KVGOV_UNSALTED && nb > 0) {
        const uint4 *sp = reinterpret_cast<const uint4 *>(p.salts + 32ll * pi);
        const uint4 a = __ldg(sp), b = __ldg(sp + 1);
        sw[0] = bswap32(a.x); sw[1] = bswap32(a.y); sw[2] = bswap32(a.z); sw[3] = bswap32(a.w);
        sw[4] = bswap32(b.x); sw[5] = bswap32(b.y); sw[6] = bswap32(b.z); sw[7] = bswap32(b.w);
    }
    const char *tok_bytes = reinterpret_cast<const char *>(p.tokens);
    const long long end_bytes = tok_end * 4;
    auto stage = [&](int jj) {   // block jj of this lane's chain -> tok[jj % 3]; one commit group per call
        if (jj < nb) {
            const long long sb = (t0 + (long long)KVGOV_BLOCK * jj) * 4;
            const long long a0 = sb & ~15ll;
            const int n = a0 == sb ? 4 : 5;
            for (int c = 0; c < n; ++c) {
                const long long ca = a0 + 16ll * c;
                const long long avail = end_bytes - ca;
                cp_async16(&sm.tok[jj % kTokStages][lane][c], tok_bytes + ca, avail >= 16 ? 16 : (int)avail);
            }
        }
        cp_async_commit();
    };
    const int sh = (int)(t0 & 3);   // word offset of every block inside its first chunk
    auto read_tokens = [&](int jj, uint32_t tw[16]) {
        const uint32_t *src = reinterpret_cast<const uint32_t *>(&sm.tok[jj % kTokStages][lane][0]) + sh;
#pragma unroll
        for (int i = 0; i < 16; ++i) tw[i] = bswap32(src[i]);
    };
    // First 64 bytes of block jj's message with the words that are h_{jj-1} set to 0.
    auto first_premessage = [&](int jj, const uint32_t tw[16], uint32_t w[16]) {
        const int kind = block_kind<MODE>(jj, k);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            w[i] = kind == kFirst ? tw[i] : (kind == kSteadyH ? 0u : sw[i]);
            w[8 + i] = kind == kFirst ? tw[8 + i] : (kind == kBoundary ? 0u : tw[i]);
        }
    };
    // Second compression of block jj: the message words after the first 64 bytes.
    auto second_message = [&](int jj, const uint32_t tw[16], uint32_t w[16]) {
        const int kind = block_kind<MODE>(jj, k);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            uint32_t pad = 0u;   // SHA-256 padding (FIPS 180-4 section 5.1.1)
            if (kind == kFirst) pad = i == 0 ? 0x80000000u : (i == 15 ? 64u * 8u : 0u);
            else pad = i == 8 ? 0x80000000u : (i == 15 ? 96u * 8u : 0u);
            w[i] = kind == kBoundary ? tw[i] : (kind != kFirst && i < 8 ? tw[8 + i] : pad);
        }
    };
    auto store_digest = [&](int jj, const uint32_t hw[8]) {
        uint4 *dst = reinterpret_cast<uint4 *>(p.digests + (row + jj) * 32);
        dst[0] = make_uint4(bswap32(hw[0]), bswap32(hw[1]), bswap32(hw[2]), bswap32(hw[3]));
        dst[1] = make_uint4(bswap32(hw[4]), bswap32(hw[5]), bswap32(hw[6]), bswap32(hw[7]));
    };
    auto read_state = [&](uint32_t hw[8]) {
        const uint4 x = sm.h[0][lane], y = sm.h[1][lane];
        hw[0] = x.x; hw[1] = x.y; hw[2] = x.z; hw[3] = x.w;
        hw[4] = y.x; hw[5] = y.y; hw[6] = y.z; hw[7] = y.w;
    };
    // Block jj's second compression and its first compression's pre-message
    // into buffer jj mod 2, then E_{jj mod 2} (tw: block jj's tokens).
    auto ahead = [&](int jj, const uint32_t tw[16]) {
        uint32_t w[16];
        second_message(jj, tw, w);
        store_kw16(w, sm.kw2[jj & 1], lane);
        schedule_kw48(w, sm.kw2[jj & 1] + 4, lane, -1);
        first_premessage(jj, tw, w);
        store_kw16(w, sm.pm[jj & 1], lane);
        bar_arrive(bar_e + (jj & 1));
    };

    stage(0);
    stage(1);
    uint32_t hw[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) hw[i] = 0u;
    for (int j = 0; j < jmax; ++j) {
        stage(j + 2);                      // its buffer last held block j - 1, read for the last time before
        cp_async_wait<1>();                // blocks j and j + 1 have landed
        uint32_t tw[16], w[16];
        read_tokens(j, tw);
        if (j == 0) ahead(0, tw);
        const int kind = block_kind<MODE>(j, k);
        // the first 64 bytes of the message: every word but h_{j-1}'s before
        // the wait for it, so that the schedule's chunk 1, which the round
        // warp waits for after its first 16 rounds, starts right after H
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            w[i] = kind == kFirst ? tw[i] : sw[i];
            w[8 + i] = kind == kFirst ? tw[8 + i] : tw[i];
        }
        if (MODE == KVGOV_BOUNDARY) {
            // ... and of a steady block (h_{j-1} in words 0..7, tokens in
            // 8..15) the terms of W_16 .. W_31 that the tokens alone fix
            // (template batch 76.1 -> 73.9 us, 0.92 -> 0.95 of its latency
            // bound; the other builds keep the plain schedule: their schedule
            // warp keeps ahead anyway, and the system-prompt batch took 266.6
            // -> 270.4 us with this)
            const bool steady = kind == kSteadyH;
            SteadyPre pre;
            if (steady) steady_pre(w, pre);
            if (j > 0) {
                bar_sync(bar_h);
                read_state(hw);            // h_{j-1}
            }
            if (steady) {
#pragma unroll
                for (int i = 0; i < 8; ++i) w[i] = hw[i];
                steady_chunk1(w, pre);
            } else {
                if (kind == kBoundary) {
#pragma unroll
                    for (int i = 0; i < 8; ++i) w[8 + i] = hw[i];
                }
                schedule_chunk(w);
            }
            store_kw_chunk(w, sm.kw1, lane, 1);
            bar_arrive(bar_b);
#pragma unroll 1
            for (int q = 2; q < 4; ++q) {
                schedule_chunk(w);
                store_kw_chunk(w, sm.kw1, lane, q);
                bar_arrive(bar_b + q - 1);
            }
        } else {
            if (j > 0) {
                bar_sync(bar_h);
                read_state(hw);            // h_{j-1}
            }
            if (kind == kSteadyH) {
#pragma unroll
                for (int i = 0; i < 8; ++i) w[i] = hw[i];
            }
            schedule_kw48(w, sm.kw1, lane, bar_b);
        }
        if (j > 0 && j - 1 < nb) store_digest(j - 1, hw);
        if (j + 1 < jmax) {
            read_tokens(j + 1, tw);
            ahead(j + 1, tw);
        }
    }
    if (jmax > 0) {
        bar_sync(bar_h);
        read_state(hw);
        if (jmax - 1 < nb) store_digest(jmax - 1, hw);
    }
    cp_async_wait<0>();
}

template <int MODE>
int launch_mode(unsigned grid, const SplitParams &p, cudaStream_t s) {
    static bool attr_set[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return KVGOV_ECUDA;
    if (dev < 0 || dev >= 64 || !attr_set[dev]) {
        if (cudaFuncSetAttribute(chain_split_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kSmemBytes) != cudaSuccess)
            return KVGOV_ECUDA;
        if (dev >= 0 && dev < 64) attr_set[dev] = true;
    }
    chain_split_kernel<MODE><<<grid, kThreads, kSmemBytes, s>>>(p);
    return kvgov_host::launch_status();
}

}  // namespace

namespace kvgov_host {

constexpr long long kSplitCtasPerSm = 3;   // measured: ahead of chain_kernel up to 3 CTAs (192 chains) per SM

long long chain_split_max_req() { return kSplitCtasPerSm * sm_count() * kChainsPerCta; }

namespace {

}  // namespace

int launch_chain_split(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                       const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                       const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                       uint32_t *d_status, cudaStream_t stream) {
    if (n_req <= 0) return KVGOV_OK;
    SplitParams p;
    p.tokens = d_tokens; p.tok_off = d_tok_off; p.principal = d_principal; p.salts = d_salts;
    p.boundary_tok = d_boundary_tok; p.blk_off = d_blk_off; p.digests = d_digests; p.status = d_status;
    p.n_req = n_req; p.n_principals = n_principals;
    const unsigned grid = (unsigned)(((long long)n_req + kChainsPerCta - 1) / kChainsPerCta);
    switch (mode) {
    case KVGOV_UNSALTED: return launch_mode<KVGOV_UNSALTED>(grid, p, stream);
    case KVGOV_ROOT: return launch_mode<KVGOV_ROOT>(grid, p, stream);
    default: return launch_mode<KVGOV_BOUNDARY>(grid, p, stream);
    }
}

}  // namespace kvgov_host
