// kvgov_chain.cu -- blocking (kvgov_block_offsets) and the chained, salted
// block digests (kvgov_chain_hash).
//
// Paper: section 2.1 equation (h_0 = H(tokens_0..B-1), h_j = H(h_{j-1},
// tokens_j)), section 4.1 equation (sigma_p prepended at the root) and
// section 4.2 equation (sigma_p prepended at the divergence block k).
//
// Chain kernel layout.  One thread owns one request's chain: the chain is
// sequential in j (each digest feeds the next message), so parallelism comes
// from the batch.  A CTA of kR threads walks block index j in lockstep; for
// every j the CTA stages the kR requests' 64-byte blocks into shared memory
// with 16-byte cp.async copies (a block starting at a token offset that is
// not a multiple of 4 spans five aligned 16-byte chunks), double-buffered so
// that the copy of block j+1 overlaps the hashing of block j.  Each thread
// then reads its 16 tokens from shared memory, byte-swaps them into
// big-endian SHA words and runs the 2 (or 3) compressions of its message in
// registers.
#include "kvgov_internal.cuh"
#include "sha256_dev.cuh"

namespace {

using namespace kvgov_dev;

// ---------------------------------------------------------------------------
// Block offsets: exclusive scan of floor(len_r / 16), three small kernels
// (tile scan, scan of tile totals, add tile bases).
// ---------------------------------------------------------------------------

constexpr int kScanThreads = 1024;
constexpr int kScanItems = 4;
constexpr int kScanTile = kScanThreads * kScanItems;

// Inclusive scan of one value per thread across a 1024-thread CTA.
__device__ __forceinline__ long long cta_inclusive_scan(long long v, long long *warp_sums) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const long long u = __shfl_up_sync(0xffffffffu, v, d);
        if (lane >= d) v += u;
    }
    if (lane == 31) warp_sums[warp] = v;
    __syncthreads();
    if (warp == 0) {
        long long s = warp_sums[lane];
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const long long u = __shfl_up_sync(0xffffffffu, s, d);
            if (lane >= d) s += u;
        }
        warp_sums[lane] = s;
    }
    __syncthreads();
    if (warp > 0) v += warp_sums[warp - 1];
    return v;
}

// Tile c covers requests [c*T, min((c+1)*T, n)).  Writes the tile-local
// inclusive counts to blk_off[r+1]; blk_off[0] = 0.
__global__ void __launch_bounds__(kScanThreads) blkoff_tile_kernel(const int64_t *__restrict__ tok_off, int32_t n,
                                                                   int64_t *__restrict__ blk_off, uint32_t *status) {
    __shared__ long long warp_sums[32];
    const long long base = (long long)blockIdx.x * kScanTile + (long long)threadIdx.x * kScanItems;
    long long cnt[kScanItems];
    long long sum = 0;
    bool bad = false;
#pragma unroll
    for (int q = 0; q < kScanItems; ++q) {
        const long long r = base + q;
        cnt[q] = 0;
        if (r < n) {
            const long long len = tok_off[r + 1] - tok_off[r];
            if (len < 0) bad = true;
            else cnt[q] = len / KVGOV_BLOCK;
        }
        sum += cnt[q];
    }
    if (bad) raise_flag(status, KVGOV_F_BADINDEX);
    long long run = cta_inclusive_scan(sum, warp_sums) - sum;
#pragma unroll
    for (int q = 0; q < kScanItems; ++q) {
        const long long r = base + q;
        run += cnt[q];
        if (r < n) blk_off[r + 1] = run;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) blk_off[0] = 0;
}

// One CTA: turn the tile totals at positions min((c+1)*T, n) into global
// inclusive prefixes.
__global__ void __launch_bounds__(kScanThreads) blkoff_carry_kernel(int32_t n, int64_t *__restrict__ blk_off) {
    __shared__ long long warp_sums[32];
    const long long n_tiles = ((long long)n + kScanTile - 1) / kScanTile;
    long long carry = 0;
    for (long long c0 = 0; c0 < n_tiles; c0 += kScanThreads) {
        const long long c = c0 + threadIdx.x;
        long long end = 0, v = 0;
        if (c < n_tiles) {
            end = (c + 1) * kScanTile;
            if (end > n) end = n;
            v = blk_off[end];
        }
        const long long inc = cta_inclusive_scan(v, warp_sums);
        const long long total = warp_sums[31];
        if (c < n_tiles) blk_off[end] = carry + inc;
        carry += total;
        __syncthreads();   // warp_sums is rewritten by the next round
    }
}

// Add the global base of tile c (now at blk_off[c*T]) to the tile's interior.
__global__ void __launch_bounds__(kScanThreads) blkoff_add_kernel(int32_t n, int64_t *__restrict__ blk_off) {
    const long long c = blockIdx.x + 1;
    const long long lo = c * kScanTile;
    long long hi = lo + kScanTile;
    if (hi > n) hi = n;
    const long long add = blk_off[lo];
    for (long long p = lo + 1 + threadIdx.x; p < hi; p += kScanThreads) blk_off[p] += add;
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
};

// Big-endian words of principal pi's 32-byte salt.
__device__ __forceinline__ void load_salt(const uint8_t *salts, int pi, uint32_t sw[8]) {
    const uint4 *s = reinterpret_cast<const uint4 *>(salts + 32ll * pi);
    const uint4 a = __ldg(s), b = __ldg(s + 1);
    sw[0] = bswap32(a.x); sw[1] = bswap32(a.y); sw[2] = bswap32(a.z); sw[3] = bswap32(a.w);
    sw[4] = bswap32(b.x); sw[5] = bswap32(b.y); sw[6] = bswap32(b.z); sw[7] = bswap32(b.w);
}

template <int MODE>
__global__ void __launch_bounds__(kR) chain_kernel(const ChainParams p) {
    __shared__ __align__(16) uint32_t stage[kStages][kR * kSlotWords];
    __shared__ long long s_tok[kR];
    __shared__ int s_nb[kR];
    __shared__ int s_jmax;

    const int tid = threadIdx.x;
    const long long r = (long long)blockIdx.x * kR + tid;
    if (tid == 0) s_jmax = 0;

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
    s_tok[tid] = nb > 0 ? t0 : 0;
    s_nb[tid] = nb;
    __syncthreads();
    if (nb > 0) atomicMax(&s_jmax, nb);
    __syncthreads();
    const int jmax = s_jmax;

    // Stage block jj of every request of the CTA into buffer buf.
    const char *tok_bytes = reinterpret_cast<const char *>(p.tokens);
    const long long end_bytes = tok_end * 4;
    auto issue = [&](int jj, int buf) {
        for (int idx = tid; idx < kR * kChunks; idx += kR) {
            const int q = idx / kChunks, c = idx - q * kChunks;
            if (jj >= s_nb[q]) continue;
            const long long sb = (s_tok[q] + (long long)KVGOV_BLOCK * jj) * 4;
            const long long a0 = sb & ~15ll;
            if (c == kChunks - 1 && a0 == sb) continue;   // aligned block: four chunks
            const long long ca = a0 + 16ll * c;
            const long long avail = end_bytes - ca;
            const int nbytes = avail >= 16 ? 16 : (int)avail;   // > 0 for every needed chunk
            cp_async16(&stage[buf][q * kSlotWords + c * 4], tok_bytes + ca, nbytes);
        }
    };

#pragma unroll
    for (int s = 0; s < kStages - 1; ++s) {
        if (s < jmax) issue(s, s);
        cp_async_commit();
    }

    const int sh = (int)(t0 & 3);   // word offset of the block inside its first chunk
    uint32_t h[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) h[i] = 0u;

    for (int j = 0; j < jmax; ++j) {
        const int jn = j + kStages - 1;
        if (jn < jmax) issue(jn, jn % kStages);
        cp_async_commit();
        cp_async_wait<kStages - 1>();
        __syncthreads();

        if (j < nb) {
            const uint32_t *src = &stage[j % kStages][tid * kSlotWords + sh];
            uint32_t tw[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) tw[i] = bswap32(src[i]);

            if (MODE == KVGOV_UNSALTED) {
                if (j == 0) sha256_msg64(tw, h);
                else sha256_msg96(h, tw, h);
            } else if (MODE == KVGOV_ROOT) {
                uint32_t pw[8];
                if (j == 0) load_salt(p.salts, pi, pw);
                else {
#pragma unroll
                    for (int i = 0; i < 8; ++i) pw[i] = h[i];
                }
                sha256_msg96(pw, tw, h);
            } else {
                if (j == k && j > 0) {
                    uint32_t sw[8];
                    load_salt(p.salts, pi, sw);
                    sha256_msg128(sw, h, tw, h);
                } else if (j == 0 && k != 0) {
                    sha256_msg64(tw, h);
                } else {
                    uint32_t pw[8];
                    if (j == k) load_salt(p.salts, pi, pw);
                    else {
#pragma unroll
                        for (int i = 0; i < 8; ++i) pw[i] = h[i];
                    }
                    sha256_msg96(pw, tw, h);
                }
            }

            uint4 *dst = reinterpret_cast<uint4 *>(p.digests + (row + j) * 32);
            dst[0] = make_uint4(bswap32(h[0]), bswap32(h[1]), bswap32(h[2]), bswap32(h[3]));
            dst[1] = make_uint4(bswap32(h[4]), bswap32(h[5]), bswap32(h[6]), bswap32(h[7]));
        }
        __syncthreads();
    }
    cp_async_wait<0>();
}

}  // namespace

extern "C" int kvgov_block_offsets(const int64_t *d_tok_off, int32_t n_req, int64_t *d_blk_off,
                                   uint32_t *d_status, kvgov_stream_t stream) {
    if (n_req < 0 || !d_tok_off || !d_blk_off) return KVGOV_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const long long n_tiles = n_req == 0 ? 1 : ((long long)n_req + kScanTile - 1) / kScanTile;
    blkoff_tile_kernel<<<(unsigned)n_tiles, kScanThreads, 0, s>>>(d_tok_off, n_req, d_blk_off, d_status);
    if (n_tiles > 1) {
        blkoff_carry_kernel<<<1, kScanThreads, 0, s>>>(n_req, d_blk_off);
        blkoff_add_kernel<<<(unsigned)(n_tiles - 1), kScanThreads, 0, s>>>(n_req, d_blk_off);
    }
    return kvgov_host::launch_status();
}

extern "C" int kvgov_chain_hash(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                                const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                                uint32_t *d_status, kvgov_stream_t stream) {
    using kvgov_host::aligned16;
    if (mode != KVGOV_UNSALTED && mode != KVGOV_ROOT && mode != KVGOV_BOUNDARY) return KVGOV_EINVAL;
    if (n_req < 0) return KVGOV_EINVAL;
    if (!d_tokens || !aligned16(d_tokens) || !d_tok_off || !d_blk_off || !d_digests || !aligned16(d_digests))
        return KVGOV_EINVAL;
    if (mode != KVGOV_UNSALTED && (!d_principal || !d_salts || !aligned16(d_salts) || n_principals <= 0))
        return KVGOV_EINVAL;
    if (mode == KVGOV_BOUNDARY && !d_boundary_tok) return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;

    ChainParams p;
    p.tokens = d_tokens; p.tok_off = d_tok_off; p.principal = d_principal; p.salts = d_salts;
    p.boundary_tok = d_boundary_tok; p.blk_off = d_blk_off; p.digests = d_digests; p.status = d_status;
    p.n_req = n_req; p.n_principals = n_principals;
    const unsigned grid = (unsigned)(((long long)n_req + kR - 1) / kR);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    switch (mode) {
    case KVGOV_UNSALTED: chain_kernel<KVGOV_UNSALTED><<<grid, kR, 0, s>>>(p); break;
    case KVGOV_ROOT: chain_kernel<KVGOV_ROOT><<<grid, kR, 0, s>>>(p); break;
    default: chain_kernel<KVGOV_BOUNDARY><<<grid, kR, 0, s>>>(p); break;
    }
    return kvgov_host::launch_status();
}
