// kvgov_blkoff.cu -- blocking (kvgov_block_offsets).
//
// Paper: section 2.1 (a request's keys are its full B-token blocks; a partial
// tail is not keyed), so request r owns floor(len_r / 16) consecutive digest
// rows starting at blk_off[r], the exclusive prefix sum of those counts.
#include "kvgov_internal.cuh"

namespace {

using namespace kvgov_dev;

// ---------------------------------------------------------------------------
// Block offsets: exclusive scan of floor(len_r / 16) in two ordinary
// launches of small CTAs, so that the scan can run in the room other kernels
// leave on the SMs (a serving pipeline runs it beside the previous batch's
// chain hash).  The n requests are cut into C <= kMaxChunks chunks of `per`
// consecutive requests.
//
//   blkoff_total_kernel   CTA c sums its chunk and posts ~total (a negative
//                         number) at blk_off[hi_c], the entry of its last
//                         request, which only CTA c writes in the next launch.
//   blkoff_scan_kernel    CTA c reads the mailboxes of the chunks before it in
//                         one round.  A mailbox holds either ~total of its
//                         chunk (posted by the first launch) or, once its CTA
//                         has finished this launch, the final inclusive prefix
//                         (>= 0).  The base of chunk c is the nearest final
//                         prefix plus the totals after it, so no CTA ever
//                         waits for another.  It then rescans its chunk and
//                         writes base + running count.
// ---------------------------------------------------------------------------

constexpr int kScanThreads = 256;
constexpr int kWarps = kScanThreads / 32;
constexpr int kMaxChunks = 1024;
constexpr int kBoxesPerThread = kMaxChunks / kScanThreads;

// Inclusive scan of one value per thread across the CTA; also returns the CTA
// total through *total.
__device__ __forceinline__ long long cta_inclusive_scan(long long v, long long *warp_sums, long long *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const long long u = __shfl_up_sync(0xffffffffu, v, d);
        if (lane >= d) v += u;
    }
    if (lane == 31) warp_sums[warp] = v;
    __syncthreads();
    if (warp == 0) {
        long long s = lane < kWarps ? warp_sums[lane] : 0;
#pragma unroll
        for (int d = 1; d < kWarps; d <<= 1) {
            const long long u = __shfl_up_sync(0xffffffffu, s, d);
            if (lane >= d) s += u;
        }
        if (lane < kWarps) warp_sums[lane] = s;
    }
    __syncthreads();
    if (warp > 0) v += warp_sums[warp - 1];
    *total = warp_sums[kWarps - 1];
    __syncthreads();   // warp_sums is reused by the next call
    return v;
}

// Largest value over the CTA.
__device__ __forceinline__ long long cta_max(long long v, long long *warp_vals) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
        const long long u = __shfl_xor_sync(0xffffffffu, v, d);
        v = u > v ? u : v;
    }
    if (lane == 0) warp_vals[warp] = v;
    __syncthreads();
    v = warp_vals[0];
#pragma unroll
    for (int w = 1; w < kWarps; ++w) v = warp_vals[w] > v ? warp_vals[w] : v;
    __syncthreads();   // warp_vals is reused by the next call
    return v;
}

__device__ __forceinline__ long long blocks_of(const int64_t *tok_off, long long r, bool *bad) {
    const long long len = tok_off[r + 1] - tok_off[r];
    if (len < 0) { *bad = true; return 0; }
    return len / KVGOV_BLOCK;
}

__device__ __forceinline__ long long chunk_end(long long c, long long per, long long n) {
    const long long e = (c + 1) * per;
    return e < n ? e : n;
}

__global__ void __launch_bounds__(kScanThreads) blkoff_total_kernel(const int64_t *__restrict__ tok_off, int32_t n,
                                                                    int64_t *blk_off, uint32_t *status,
                                                                    long long per) {
    __shared__ long long warp_sums[kWarps];
    const long long lo = (long long)blockIdx.x * per, hi = chunk_end(blockIdx.x, per, n);
    bool bad = false;
    long long part = 0;
    for (long long r = lo + threadIdx.x; r < hi; r += kScanThreads) part += blocks_of(tok_off, r, &bad);
    long long total;
    cta_inclusive_scan(part, warp_sums, &total);
    if (threadIdx.x == 0 && hi > lo) blk_off[hi] = ~total;
    if (bad) raise_flag(status, KVGOV_F_BADINDEX);
}

__global__ void __launch_bounds__(kScanThreads) blkoff_scan_kernel(const int64_t *__restrict__ tok_off, int32_t n,
                                                                   int64_t *blk_off, long long per) {
    __shared__ long long warp_sums[kWarps];
    const long long c = blockIdx.x;
    const long long lo = c * per, hi = chunk_end(c, per, n);

    // the mailboxes of chunks t < c: ~total (< 0) or the final prefix (>= 0)
    long long box[kBoxesPerThread];
    long long nearest = -1;
#pragma unroll
    for (int k = 0; k < kBoxesPerThread; ++k) {
        const long long t = threadIdx.x + (long long)k * kScanThreads;
        box[k] = 0;
        if (t < c) {
            box[k] = (long long)__ldcg(reinterpret_cast<const unsigned long long *>(blk_off) + chunk_end(t, per, n));
            if (box[k] >= 0) nearest = t;
        }
    }
    nearest = cta_max(nearest, warp_sums);
    long long add = 0;
#pragma unroll
    for (int k = 0; k < kBoxesPerThread; ++k) {
        const long long t = threadIdx.x + (long long)k * kScanThreads;
        if (t < c && t > nearest) add += ~box[k];
        if (t == nearest) add += box[k];
    }
    long long base;
    cta_inclusive_scan(add, warp_sums, &base);

    if (c == 0 && threadIdx.x == 0) blk_off[0] = 0;
    long long carry = base;
    for (long long r0 = lo; r0 < hi; r0 += kScanThreads) {
        const long long r = r0 + threadIdx.x;
        bool ignored = false;
        const long long cnt = r < hi ? blocks_of(tok_off, r, &ignored) : 0;
        long long chunk;
        const long long inc = cta_inclusive_scan(cnt, warp_sums, &chunk);
        if (r < hi) blk_off[r + 1] = carry + inc;
        carry += chunk;
    }
}

}  // namespace

extern "C" int kvgov_block_offsets(const int64_t *d_tok_off, int32_t n_req, int64_t *d_blk_off,
                                   uint32_t *d_status, kvgov_stream_t stream) {
    if (n_req < 0 || !d_tok_off || !d_blk_off) return KVGOV_EINVAL;
    const long long n = n_req;
    const long long per_min = (n + kMaxChunks - 1) / kMaxChunks;
    const long long per = per_min > kScanThreads ? per_min : kScanThreads;
    const long long chunks = (n + per - 1) / per;
    const unsigned grid = chunks > 0 ? (unsigned)chunks : 1u;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (chunks > 0) blkoff_total_kernel<<<grid, kScanThreads, 0, s>>>(d_tok_off, n_req, d_blk_off, d_status, per);
    blkoff_scan_kernel<<<grid, kScanThreads, 0, s>>>(d_tok_off, n_req, d_blk_off, per);
    return kvgov_host::launch_status();
}

extern "C" int kvgov_count_blocks(const int64_t *h_tok_off, int32_t n_req, int64_t *h_blk_off, int64_t *n_blocks) {
    if (n_req < 0 || !h_tok_off || !n_blocks) return KVGOV_EINVAL;
    // floor(len_r / 16) per request, a negative length counting 0, as
    // blocks_of does on the device
    long long total = 0;
    if (h_blk_off) h_blk_off[0] = 0;
    for (int32_t r = 0; r < n_req; ++r) {
        const long long len = h_tok_off[r + 1] - h_tok_off[r];
        total += len < 0 ? 0 : len / KVGOV_BLOCK;
        if (h_blk_off) h_blk_off[r + 1] = total;
    }
    *n_blocks = total;
    return KVGOV_OK;
}
