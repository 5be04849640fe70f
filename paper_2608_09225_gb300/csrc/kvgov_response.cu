// kvgov_response.cu -- exact-response cache keys (kvgov_response_key).
//
// Paper: Table 1 (an exact-response cache keys on byte equality of the whole
// prompt) and section 4.1 (that cache is isolated by prepending sigma_p to
// its key).  The key of request r is SHA-256(sigma_p || prompt bytes), or
// SHA-256(prompt bytes) unsalted: one message per request, every token
// included (no block truncation), with the FIPS 180-4 padding after it.
//
// Layout as in the chain kernel: one thread per request, kR requests per
// CTA, each thread staging its own request's 64-byte token blocks into
// shared memory with 16-byte cp.async copies, double-buffered, with no
// barrier between blocks (a warp walks its longest message).  The message
// stream is the salt's 8 words (salted) followed by the big-endian token
// words, so with a salt a message block is the last 8 words of token block
// m-1 (kept in registers) and the first 8 of token block m.  Words past the
// prompt become the padding: 0x80000000, zeros, and in the last message
// block the 64-bit bit length.
//
// A batch too small to fill the GPU (at most kvgov_host::chain_split_max_req()
// requests) runs response_split_kernel instead: one request's message is
// sequential in its blocks, so such a batch leaves each SM sub-partition one
// warp at most, and a warp alone there is bound by the latency of its own
// instructions.  Per 32 requests a round warp runs only the 64 rounds of each
// compression, reading K_t + W_t from shared memory, and a schedule warp on
// another sub-partition stages the tokens, builds each message block and
// expands its schedule; no schedule depends on the running state, so the
// schedule warp fills a ring of two buffers ahead of the round warp (named
// barriers FULL_b: buffer b filled; EMPTY_b: buffer b read and free).
#include "kvgov_internal.cuh"
#include "kvgov_split.cuh"
#include "sha256_dev.cuh"

namespace {

using namespace kvgov_dev;

constexpr int kR = 128;           // requests (threads) per CTA
constexpr int kStages = 2;
constexpr int kChunks = 5;        // 16-byte chunks that can cover one 64-byte block
constexpr int kSlotWords = kChunks * 4;

struct ResponseParams {
    const int32_t *tokens;
    const int64_t *tok_off;
    const int32_t *principal;
    const uint8_t *salts;
    uint8_t *keys;
    uint32_t *status;
    int32_t n_req;
    int32_t n_principals;
};

template <bool SALTED>
__global__ void __launch_bounds__(kR) response_key_kernel(const ResponseParams p) {
    __shared__ __align__(16) uint32_t stage[kStages][kR * kSlotWords];

    constexpr int S = SALTED ? 8 : 0;        // salt words ahead of the prompt
    const int tid = threadIdx.x;
    const long long r = (long long)blockIdx.x * kR + tid;

    const long long tok_end = p.tok_off[p.n_req];
    long long t0 = 0, len = 0;
    int nbt = 0, nmsg = 0, pi = 0;
    if (r < p.n_req) {
        t0 = p.tok_off[r];
        const long long t1 = p.tok_off[r + 1];
        len = t1 - t0;
        bool ok = t0 >= 0 && t1 >= t0 && t1 <= tok_end && len < (1ll << 28);
        if (SALTED) {
            pi = p.principal[r];
            ok = ok && pi >= 0 && pi < p.n_principals;
        }
        if (ok) {
            nbt = (int)((len + KVGOV_BLOCK - 1) / KVGOV_BLOCK);
            nmsg = (int)((S + len + 3 + 15) / 16);
        } else {
            raise_flag(p.status, KVGOV_F_BADINDEX);
            len = 0;
        }
    }
    // Each thread stages and reads only its own request's blocks: no barrier
    // between message blocks, and a warp walks its own longest message.
    const int mmax = (int)__reduce_max_sync(0xffffffffu, (unsigned)nmsg);

    const char *tok_bytes = reinterpret_cast<const char *>(p.tokens);
    const long long end_bytes = tok_end * 4;
    auto issue = [&](int jj, int buf) {        // this thread's request's token block jj (as the chain kernel)
        if (jj < nbt) {
            const long long sb = (t0 + (long long)KVGOV_BLOCK * jj) * 4;
            const long long a0 = sb & ~15ll;
#pragma unroll
            for (int c = 0; c < kChunks; ++c) {
                if (c == kChunks - 1 && a0 == sb) break;      // aligned block: four chunks
                const long long ca = a0 + 16ll * c;
                const long long avail = end_bytes - ca;
                if (avail <= 0) break;                         // a partial last block at the end of the array
                cp_async16(&stage[buf][tid * kSlotWords + c * 4], tok_bytes + ca, avail >= 16 ? 16 : (int)avail);
            }
        }
    };
#pragma unroll
    for (int s = 0; s < kStages - 1; ++s) {
        if (s < mmax) issue(s, s);
        cp_async_commit();
    }

    const AddAlu add{};
    const int sh = (int)(t0 & 3);
    uint32_t st[8];
    sha_iv(st);
    uint32_t carry[8];                          // salted: the stream words before this block's tokens
    if (SALTED && nmsg > 0) {
        const uint4 *s = reinterpret_cast<const uint4 *>(p.salts + 32ll * pi);
        const uint4 a = __ldg(s), b = __ldg(s + 1);
        carry[0] = bswap32(a.x); carry[1] = bswap32(a.y); carry[2] = bswap32(a.z); carry[3] = bswap32(a.w);
        carry[4] = bswap32(b.x); carry[5] = bswap32(b.y); carry[6] = bswap32(b.z); carry[7] = bswap32(b.w);
    } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) carry[i] = 0u;
    }
    const unsigned long long bits = (unsigned long long)(4 * S + 4 * len) * 8ull;
    const long long end_word = S + len;         // stream index of the 0x80000000 word

    for (int m = 0; m < mmax; ++m) {
        const int jn = m + kStages - 1;
        if (jn < mmax) issue(jn, jn % kStages);
        cp_async_commit();
        cp_async_wait<kStages - 1>();      // this thread's copies of block m have landed

        if (m < nmsg) {
            const uint32_t *src = &stage[m % kStages][tid * kSlotWords + sh];
            uint32_t tw[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) tw[i] = bswap32(src[i]);   // stale past the prompt: masked below
            uint32_t w[16];
            if (16ll * m + 15 < end_word) {                         // every word is the prompt's
#pragma unroll
                for (int i = 0; i < 16; ++i) w[i] = SALTED ? (i < 8 ? carry[i] : tw[i - 8]) : tw[i];
            } else {
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const uint32_t v = SALTED ? (i < 8 ? carry[i] : tw[i - 8]) : tw[i];
                    const long long k = 16ll * m + i;               // stream word index
                    w[i] = k < end_word ? v : (k == end_word ? 0x80000000u : 0u);
                }
            }
            if (SALTED) {
#pragma unroll
                for (int i = 0; i < 8; ++i) carry[i] = tw[i + 8];
            }
            if (m == nmsg - 1) {
                w[14] = (uint32_t)(bits >> 32);
                w[15] = (uint32_t)bits;
            }
            sha_compress_small(st, w, add);
        }
    }
    cp_async_wait<0>();
    if (r < p.n_req) {
        uint4 *dst = reinterpret_cast<uint4 *>(p.keys + 32 * r);
        dst[0] = make_uint4(bswap32(st[0]), bswap32(st[1]), bswap32(st[2]), bswap32(st[3]));
        dst[1] = make_uint4(bswap32(st[4]), bswap32(st[5]), bswap32(st[6]), bswap32(st[7]));
    }
}

// Shared memory of one round/schedule pair of response_split_kernel.
constexpr int kSplitPairs = 2;
constexpr int kSplitThreads = 64 * kSplitPairs;
constexpr int kSplitReqPerCta = 32 * kSplitPairs;
constexpr int kTokStages = 3;       // token blocks m, m + 1 and m + 2 in flight
struct ResponsePairSmem {
    uint4 kw[2][16][32];            // K_t + W_t of message blocks m, m + 1 (by parity)
    uint4 tok[kTokStages][32][kChunks];
};

template <bool SALTED>
__global__ void __launch_bounds__(kSplitThreads, 1) response_split_kernel(const ResponseParams p) {
    __shared__ ResponsePairSmem smem[kSplitPairs];
    constexpr int S = SALTED ? 8 : 0;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int pair = warp >> 1;
    const bool round_warp = (warp & 1) == 0;
    ResponsePairSmem &sm = smem[pair];
    const int bar_full = 1 + 4 * pair, bar_empty = bar_full + 2;

    // Per-request set-up (both warps of the pair hold the same request in the same lane).
    const long long r = (long long)blockIdx.x * kSplitReqPerCta + pair * 32 + lane;
    const long long tok_end = p.tok_off[p.n_req];
    long long t0 = 0, len = 0;
    int nbt = 0, nmsg = 0, pi = 0;
    if (r < p.n_req) {
        t0 = p.tok_off[r];
        const long long t1 = p.tok_off[r + 1];
        len = t1 - t0;
        bool ok = t0 >= 0 && t1 >= t0 && t1 <= tok_end && len < (1ll << 28);
        if (SALTED) {
            pi = p.principal[r];
            ok = ok && pi >= 0 && pi < p.n_principals;
        }
        if (ok) {
            nbt = (int)((len + KVGOV_BLOCK - 1) / KVGOV_BLOCK);
            nmsg = (int)((S + len + 3 + 15) / 16);
        } else {
            if (!round_warp) raise_flag(p.status, KVGOV_F_BADINDEX);
            len = 0;
        }
    }
    const int mmax = (int)__reduce_max_sync(0xffffffffu, (unsigned)nmsg);   // the same in both warps

    if (round_warp) {
        uint32_t st[8], v[8], ka[16], kb[16];
        sha_iv(st);
        for (int m = 0; m < mmax; ++m) {
            bar_sync(bar_full + (m & 1));
            const uint4 (*kw)[32] = sm.kw[m & 1];
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] = st[i];
            load16(kw, lane, ka);
#pragma unroll 1
            for (int q = 0; q < 4; q += 2) {   // each chunk's values load while the previous chunk's rounds run
                load16(kw + 4 * (q + 1), lane, kb);
                sha_rounds16_t1t2(v, ka);
                if (q + 2 < 4) load16(kw + 4 * (q + 2), lane, ka);
                sha_rounds16_t1t2(v, kb);
            }
            if (m + 2 < mmax) bar_arrive(bar_empty + (m & 1));   // the buffer is read: free for message m + 2
            if (m < nmsg) {
#pragma unroll
                for (int i = 0; i < 8; ++i) st[i] += v[i];
            }
        }
        if (r < p.n_req) {
            uint4 *dst = reinterpret_cast<uint4 *>(p.keys + 32 * r);
            dst[0] = make_uint4(bswap32(st[0]), bswap32(st[1]), bswap32(st[2]), bswap32(st[3]));
            dst[1] = make_uint4(bswap32(st[4]), bswap32(st[5]), bswap32(st[6]), bswap32(st[7]));
        }
        return;
    }

    // Schedule warp.
    uint32_t carry[8];   // salted: the stream words before this block's tokens
    if (SALTED && nmsg > 0) {
        const uint4 *s = reinterpret_cast<const uint4 *>(p.salts + 32ll * pi);
        const uint4 a = __ldg(s), b = __ldg(s + 1);
        carry[0] = bswap32(a.x); carry[1] = bswap32(a.y); carry[2] = bswap32(a.z); carry[3] = bswap32(a.w);
        carry[4] = bswap32(b.x); carry[5] = bswap32(b.y); carry[6] = bswap32(b.z); carry[7] = bswap32(b.w);
    } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) carry[i] = 0u;
    }
    const char *tok_bytes = reinterpret_cast<const char *>(p.tokens);
    const long long end_bytes = tok_end * 4;
    auto stage = [&](int jj) {   // token block jj of this lane's request -> tok[jj % 3]; one commit group per call
        if (jj < nbt) {
            const long long sb = (t0 + (long long)KVGOV_BLOCK * jj) * 4;
            const long long a0 = sb & ~15ll;
            const int n = a0 == sb ? 4 : 5;
            for (int c = 0; c < n; ++c) {
                const long long ca = a0 + 16ll * c;
                const long long avail = end_bytes - ca;
                if (avail <= 0) break;            // a partial last block at the end of the array
                cp_async16(&sm.tok[jj % kTokStages][lane][c], tok_bytes + ca, avail >= 16 ? 16 : (int)avail);
            }
        }
        cp_async_commit();
    };
    const int sh = (int)(t0 & 3);
    const unsigned long long bits = (unsigned long long)(4 * S + 4 * len) * 8ull;
    const long long end_word = S + len;       // stream index of the 0x80000000 word
    stage(0);
    stage(1);
    for (int m = 0; m < mmax; ++m) {
        stage(m + 2);                         // its buffer last held token block m - 1, read in iteration m - 1
        cp_async_wait<1>();                   // token blocks m and m + 1 have landed
        const uint32_t *src = reinterpret_cast<const uint32_t *>(&sm.tok[m % kTokStages][lane][0]) + sh;
        uint32_t tw[16], w[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) tw[i] = bswap32(src[i]);   // stale past the prompt: masked below
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const uint32_t x = SALTED ? (i < 8 ? carry[i] : tw[i - 8]) : tw[i];
            const long long k = 16ll * m + i;                   // stream word index
            w[i] = k < end_word ? x : (k == end_word ? 0x80000000u : 0u);
        }
        if (SALTED) {
#pragma unroll
            for (int i = 0; i < 8; ++i) carry[i] = tw[i + 8];
        }
        if (m == nmsg - 1) {
            w[14] = (uint32_t)(bits >> 32);
            w[15] = (uint32_t)bits;
        }
        if (m >= 2) bar_sync(bar_empty + (m & 1));   // message m - 2 has been read from this buffer
        store_kw16(w, sm.kw[m & 1], lane);
        schedule_kw48(w, sm.kw[m & 1] + 4, lane, -1);
        bar_arrive(bar_full + (m & 1));
    }
    cp_async_wait<0>();
}

}  // namespace

extern "C" int kvgov_response_key(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                  const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                                  uint8_t *d_keys, uint32_t *d_status, kvgov_stream_t stream) {
    using kvgov_host::aligned16;
    if (mode != KVGOV_UNSALTED && mode != KVGOV_ROOT) return KVGOV_EINVAL;
    if (n_req < 0 || !d_tok_off) return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;
    if (!d_tokens || !aligned16(d_tokens) || !d_keys || !aligned16(d_keys)) return KVGOV_EINVAL;
    if (mode == KVGOV_ROOT && (!d_principal || !d_salts || !aligned16(d_salts) || n_principals <= 0))
        return KVGOV_EINVAL;
    ResponseParams p;
    p.tokens = d_tokens; p.tok_off = d_tok_off; p.principal = d_principal; p.salts = d_salts;
    p.keys = d_keys; p.status = d_status; p.n_req = n_req; p.n_principals = n_principals;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (n_req <= kvgov_host::chain_split_max_req()) {   // a batch too small to fill the GPU: two warps per 32
        const unsigned g = (unsigned)(((long long)n_req + kSplitReqPerCta - 1) / kSplitReqPerCta);
        if (mode == KVGOV_ROOT) response_split_kernel<true><<<g, kSplitThreads, 0, s>>>(p);
        else response_split_kernel<false><<<g, kSplitThreads, 0, s>>>(p);
        return kvgov_host::launch_status();
    }
    const unsigned grid = (unsigned)(((long long)n_req + kR - 1) / kR);
    if (mode == KVGOV_ROOT) response_key_kernel<true><<<grid, kR, 0, s>>>(p);
    else response_key_kernel<false><<<grid, kR, 0, s>>>(p);
    return kvgov_host::launch_status();
}
