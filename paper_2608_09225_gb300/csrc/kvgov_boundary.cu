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
// A warp per request, or four requests per warp (8 lanes each) for batches
// of many requests.  Each round a request's lanes compare its next tokens
// (coalesced loads; the preamble's tokens read through the read-only path:
// every request of a preamble reads the same ones, so they stay in L2) and a
// ballot per load finds the first mismatch.
#include "kvgov_internal.cuh"

namespace {

using namespace kvgov_dev;

constexpr int kThreads = 256;

// The candidate preambles of a request: its own (one), none, or all.
__device__ __forceinline__ int n_candidates(int id, int n_tpl) {
    return id == KVGOV_TEMPLATE_NONE ? 0 : (id == KVGOV_TEMPLATE_ANY ? n_tpl : 1);
}

// G lanes per request (32 / G requests per warp), kPer tokens per lane per
// round: G * kPer tokens of each request compared per round.
template <int G, int kPer>
__global__ void __launch_bounds__(kThreads) boundary_kernel(const int32_t *__restrict__ tokens,
                                                            const int64_t *__restrict__ tok_off, int32_t n_req,
                                                            const int32_t *__restrict__ template_id,
                                                            const int32_t *__restrict__ tpl_tokens,
                                                            const int64_t *__restrict__ tpl_off, int32_t n_tpl,
                                                            int32_t *__restrict__ boundary_tok, uint32_t *status) {
    constexpr int kSegs = 32 / G;
    constexpr unsigned kSegMask = G == 32 ? 0xffffffffu : ((1u << G) - 1u);
    const int lane = threadIdx.x & 31, seg = lane / G, sl = lane % G;
    const long long warps_total = (long long)gridDim.x * (kThreads / 32);
    const long long tok_end = tok_off[n_req];
    const long long tpl_end = n_tpl > 0 ? tpl_off[n_tpl] : 0;
    for (long long w = ((long long)blockIdx.x * kThreads + threadIdx.x) / 32; w * kSegs < n_req;
         w += warps_total) {                                   // warp-uniform
        const long long r = w * kSegs + seg;
        long long t0 = 0, len = 0;
        int id = KVGOV_TEMPLATE_NONE;
        bool bad = false;
        if (r < n_req) {
            t0 = tok_off[r];
            const long long t1 = tok_off[r + 1];
            id = template_id[r];
            bad = t0 < 0 || t1 < t0 || t1 > tok_end || id < KVGOV_TEMPLATE_ANY || id >= n_tpl;
            len = t1 - t0;
        }
        const int ncand = (r < n_req && !bad) ? n_candidates(id, n_tpl) : 0;
        const int cmax = __reduce_max_sync(0xffffffffu, (unsigned)ncand);
        long long best = 0;
        for (int c = 0; c < cmax; ++c) {                       // warp-uniform
            // this group's c-th candidate, its length and the tokens to compare
            long long n = 0, s0 = 0;
            if (c < ncand) {
                const int t = id == KVGOV_TEMPLATE_ANY ? c : id;
                s0 = tpl_off[t];
                const long long s1 = tpl_off[t + 1];
                if (s0 < 0 || s1 < s0 || s1 > tpl_end) bad = true;
                else n = len < s1 - s0 ? len : s1 - s0;
            }
            if (n <= best) n = 0;                              // cannot beat the best so far
            const int32_t *a = tokens + t0, *b = tpl_tokens + s0;
            long long l = 0;
            bool active = n > 0;
            while (__any_sync(0xffffffffu, active)) {          // rounds of G * kPer tokens per request
                unsigned miss[kPer];
#pragma unroll
                for (int u = 0; u < kPer; ++u) {
                    const long long i = l + u * G + sl;
                    const bool differ = active && i < n && a[i] != __ldg(b + i);
                    miss[u] = G == 32 ? __ballot_sync(0xffffffffu, differ)
                                      : (__ballot_sync(0xffffffffu, differ) >> (seg * G)) & kSegMask;
                }
                if (active) {
                    long long hit = -1;
#pragma unroll
                    for (int u = kPer - 1; u >= 0; --u)
                        if (miss[u]) hit = l + u * G + __ffs((int)miss[u]) - 1;
                    if (hit >= 0) { l = hit; active = false; }
                    else {
                        l += kPer * G;
                        if (l >= n) { l = n; active = false; }
                    }
                }
            }
            if (l > best) best = l;
        }
        if (bad) best = 0;
        if (r < n_req && sl == 0) {
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
    // Batches of many requests: four requests per warp, 64 tokens each per
    // round, so more requests are in flight than the SMs hold warps.  Fewer
    // requests (which may have long preambles): a warp per request, 128 tokens
    // per round.
    const bool many = n_req >= 32 * 1024;
    const int per_warp = many ? 4 : 1;
    const long long warps = ((long long)n_req + per_warp - 1) / per_warp;
    long long grid = (warps + (kThreads / 32) - 1) / (kThreads / 32);
    const long long cap = (long long)kvgov_host::sm_count() * 32;
    if (grid > cap) grid = cap;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (many)
        boundary_kernel<8, 8><<<(unsigned)grid, kThreads, 0, s>>>(d_tokens, d_tok_off, n_req, d_template_id,
                                                                  d_tpl_tokens, d_tpl_off, n_tpl, d_boundary_tok,
                                                                  d_status);
    else
        boundary_kernel<32, 4><<<(unsigned)grid, kThreads, 0, s>>>(d_tokens, d_tok_off, n_req, d_template_id,
                                                                   d_tpl_tokens, d_tpl_off, n_tpl, d_boundary_tok,
                                                                   d_status);
    return kvgov_host::launch_status();
}
