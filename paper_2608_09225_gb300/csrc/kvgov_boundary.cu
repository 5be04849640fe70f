// kvgov_boundary.cu -- divergence-boundary detection (kvgov_divergence_boundary).
//
// Paper: section 4.2 (the salt goes in at the divergence boundary k: blocks
// before it hold the shared preamble, which carries no signal that tells
// principals apart) and section 5.7 (a divergence at token i invalidates
// every block from floor(i/B) on).  Given preambles registered by the
// operator (system prompts, form templates), a request's boundary token
// offset is the length of its longest common prefix with its preamble:
// the first token where it diverges.  kvgov_chain_hash in BOUNDARY mode then
// salts from block floor(b / 16) on.
//
// One warp per request.  Each round the warp compares the next 128 tokens
// (4 coalesced 128-byte loads of the request, the preamble's tokens read
// through the read-only path: every request of a preamble reads the same
// ones, so they stay in L2) and a ballot per load finds the first mismatch.
#include "kvgov_internal.cuh"

namespace {

using namespace kvgov_dev;

constexpr int kThreads = 256;
constexpr int kUnroll = 4;                  // 32-token loads per warp per round

// Longest common prefix of a[0..n) and b[0..n), computed by the whole warp.
__device__ __forceinline__ long long warp_lcp(const int32_t *__restrict__ a, const int32_t *__restrict__ b,
                                              long long n) {
    const int lane = threadIdx.x & 31;
    for (long long i0 = 0; i0 < n; i0 += 32 * kUnroll) {
        unsigned miss[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const long long i = i0 + 32 * u + lane;
            const bool differ = i < n && a[i] != __ldg(b + i);
            miss[u] = __ballot_sync(0xffffffffu, differ);
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
            if (miss[u]) return i0 + 32 * u + __ffs((int)miss[u]) - 1;
    }
    return n;
}

__global__ void __launch_bounds__(kThreads) boundary_kernel(const int32_t *__restrict__ tokens,
                                                            const int64_t *__restrict__ tok_off, int32_t n_req,
                                                            const int32_t *__restrict__ template_id,
                                                            const int32_t *__restrict__ tpl_tokens,
                                                            const int64_t *__restrict__ tpl_off, int32_t n_tpl,
                                                            int32_t *__restrict__ boundary_tok, uint32_t *status) {
    const int lane = threadIdx.x & 31;
    const long long warps_total = (long long)gridDim.x * (kThreads / 32);
    const long long tok_end = tok_off[n_req];
    const long long tpl_end = n_tpl > 0 ? tpl_off[n_tpl] : 0;
    for (long long r = ((long long)blockIdx.x * kThreads + threadIdx.x) / 32; r < n_req; r += warps_total) {
        const long long t0 = tok_off[r], t1 = tok_off[r + 1];
        const int id = template_id[r];
        bool bad = t0 < 0 || t1 < t0 || t1 > tok_end || id < KVGOV_TEMPLATE_ANY || id >= n_tpl;
        long long best = 0;
        if (!bad && id != KVGOV_TEMPLATE_NONE) {
            const int lo = id == KVGOV_TEMPLATE_ANY ? 0 : id;
            const int hi = id == KVGOV_TEMPLATE_ANY ? n_tpl : id + 1;
            for (int t = lo; t < hi; ++t) {                       // warp-uniform
                const long long s0 = tpl_off[t], s1 = tpl_off[t + 1];
                if (s0 < 0 || s1 < s0 || s1 > tpl_end) {
                    bad = true;
                    break;
                }
                const long long n = (t1 - t0) < (s1 - s0) ? (t1 - t0) : (s1 - s0);
                if (n <= best) continue;                           // cannot beat the best so far
                const long long l = warp_lcp(tokens + t0, tpl_tokens + s0, n);
                if (l > best) best = l;
            }
        }
        if (bad) best = 0;
        if (lane == 0) {
            boundary_tok[r] = (int32_t)best;
            if (bad) raise_flag(status, KVGOV_F_BADINDEX);
        }
    }
}

}  // namespace

extern "C" int kvgov_divergence_boundary(const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                         const int32_t *d_template_id, const int32_t *d_tpl_tokens,
                                         const int64_t *d_tpl_off, int32_t n_tpl, int32_t *d_boundary_tok,
                                         uint32_t *d_status, kvgov_stream_t stream) {
    if (n_req < 0 || n_tpl < 0 || !d_tok_off) return KVGOV_EINVAL;
    if (n_req == 0) return KVGOV_OK;
    if (!d_tokens || !d_template_id || !d_boundary_tok) return KVGOV_EINVAL;
    if (n_tpl > 0 && (!d_tpl_tokens || !d_tpl_off)) return KVGOV_EINVAL;
    long long grid = ((long long)n_req + (kThreads / 32) - 1) / (kThreads / 32);
    const long long cap = (long long)kvgov_host::sm_count() * 32;
    if (grid > cap) grid = cap;
    boundary_kernel<<<(unsigned)grid, kThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        d_tokens, d_tok_off, n_req, d_template_id, d_tpl_tokens, d_tpl_off, n_tpl, d_boundary_tok, d_status);
    return kvgov_host::launch_status();
}
