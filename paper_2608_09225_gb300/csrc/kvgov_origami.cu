// kvgov_origami.cu -- ORIGAMI audit allocation, batched (kvgov_origami).
//
// Paper: section 4.3, Theorem (ORIGAMI water-filling solution).  The defender
// spreads an audit budget K over tenants with values at risk v_i > 0 to
// minimise the adversary's best payoff max_i v_i (1 - p_i) subject to
// sum_i p_i = K, p_i in [0, 1]; the optimum is p_i = max(0, 1 - lambda / v_i)
// with the unique water level lambda meeting the budget.
//
// One warp per problem, in fp32.  The budget as a function of the level,
// f(lambda) = sum_i max(0, 1 - lambda / v_i), is decreasing, convex and
// piecewise linear, with a kink at every v_i.  Newton's method from
// lambda = 0 stays below the root and ends on it: each step takes the
// tenants still above the level (m of them, S = sum of their 1 / v_i) and
// solves f = K on that piece, lambda' = (m - K) / S; when the set above the
// new level is the same set, lambda' is the water level.  The set shrinks at
// every other step, so there are at most (number of tenants + 1) steps.  The
// paper finds lambda by bisection; this reaches the same level without an
// iteration count that sets the precision.
#include <cmath>

#include "kvgov_internal.cuh"

namespace {

using namespace kvgov_dev;

constexpr int kThreads = 256;
constexpr int kRegSlots = 4;                 // tenants per lane kept in registers

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) v += __shfl_xor_sync(0xffffffffu, v, d);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, d));
    return v;
}
__device__ __forceinline__ int warp_isum(int v) { return __reduce_add_sync(0xffffffffu, (unsigned)v); }

// A tenant takes part if its value is positive and finite; v <= 0 gets no
// audit (no payoff to protect), NaN or infinity is flagged and gets none.
__device__ __forceinline__ bool usable(float v) { return v > 0.0f && v <= 3.0e38f; }

__global__ void __launch_bounds__(kThreads) origami_kernel(const float *__restrict__ values,
                                                           const int64_t *__restrict__ off, int32_t n_prob,
                                                           const float *__restrict__ budget, float *__restrict__ p,
                                                           float *__restrict__ lambda_out,
                                                           float *__restrict__ utility_out, uint32_t *status) {
    const int lane = threadIdx.x & 31;
    const long long warps_total = (long long)gridDim.x * (kThreads / 32);
    const long long total = off[n_prob];
    for (long long q = ((long long)blockIdx.x * kThreads + threadIdx.x) / 32; q < n_prob; q += warps_total) {
        const long long b0 = off[q], b1 = off[q + 1];
        bool bad = b0 < 0 || b1 < b0 || b1 > total;
        const long long n = bad ? 0 : b1 - b0;
        const float *v = values + b0;

        // usable tenants, largest value, values that are not numbers
        int my_pos = 0, my_bad = 0;
        float my_max = 0.0f;
        for (long long i = lane; i < n; i += 32) {
            const float x = v[i];
            if (usable(x)) { ++my_pos; my_max = fmaxf(my_max, x); }
            else if (!(x <= 0.0f)) ++my_bad;          // NaN or +infinity
        }
        const int npos = warp_isum(my_pos);
        const float vmax = warp_max(my_max);
        float K = budget[q];
        if (warp_isum(my_bad) > 0 || !(K >= 0.0f)) bad = true;
        if (!(K >= 0.0f)) K = 0.0f;
        if (K > (float)npos) K = (float)npos;

        float lam;
        if (npos == 0 || K <= 0.0f) {
            lam = vmax;                                   // nothing to spend: p = 0
        } else if (K >= (float)npos) {
            lam = 0.0f;                                   // every usable tenant audited
        } else if (n <= 32 * kRegSlots) {
            // up to 128 tenants: values and their reciprocals stay in registers
            float x[kRegSlots], rx[kRegSlots];
#pragma unroll
            for (int k = 0; k < kRegSlots; ++k) {
                const long long i = lane + 32 * k;
                const float xi = i < n ? v[i] : 0.0f;
                x[k] = usable(xi) ? xi : 0.0f;            // 0: never above the level
                rx[k] = x[k] > 0.0f ? __frcp_rn(x[k]) : 0.0f;
            }
            lam = 0.0f;
            int prev_m = -1;
            for (int step = 0; step <= npos + 1; ++step) {          // warp-uniform
                float s = 0.0f;
                int m = 0;
#pragma unroll
                for (int k = 0; k < kRegSlots; ++k)
                    if (x[k] > lam) { s += rx[k]; ++m; }
                s = warp_sum(s);
                m = warp_isum(m);
                const float next = ((float)m - K) / s;
                if (m == prev_m) { lam = next; break; }
                lam = fmaxf(lam, next);
                prev_m = m;
            }
        } else {
            lam = 0.0f;
            int prev_m = -1;
            for (int step = 0; step <= npos + 1; ++step) {          // warp-uniform
                float s = 0.0f;
                int m = 0;
                for (long long i = lane; i < n; i += 32) {
                    const float x = v[i];
                    if (usable(x) && x > lam) { s += __frcp_rn(x); ++m; }
                }
                s = warp_sum(s);
                m = warp_isum(m);
                const float next = ((float)m - K) / s;
                if (m == prev_m) { lam = next; break; }
                lam = fmaxf(lam, next);
                prev_m = m;
            }
        }

        // p_i, and the adversary's payoff v_i (1 - p_i): min(v_i, lambda) for a
        // usable tenant (lambda where audited, v_i where not), written that
        // way because 1 - p_i cancels when p_i is close to 1.
        float my_u = -3.0e38f;
        for (long long i = lane; i < n; i += 32) {
            const float x = v[i];
            const float pi = usable(x) ? fmaxf(0.0f, 1.0f - lam / x) : 0.0f;
            p[b0 + i] = pi;
            if (!isnan(x)) my_u = fmaxf(my_u, usable(x) ? fminf(x, lam) : x);
        }
        const float u = warp_max(my_u);
        if (lane == 0) {
            if (lambda_out) lambda_out[q] = lam;
            if (utility_out) utility_out[q] = n > 0 ? u : 0.0f;
            if (bad) raise_flag(status, KVGOV_F_BADINDEX);
        }
    }
}

}  // namespace

extern "C" int kvgov_origami(const float *d_values, const int64_t *d_off, int32_t n_prob, const float *d_budget,
                             float *d_p, float *d_lambda, float *d_utility, uint32_t *d_status,
                             kvgov_stream_t stream) {
    if (n_prob < 0 || !d_off) return KVGOV_EINVAL;
    if (n_prob == 0) return KVGOV_OK;
    if (!d_values || !d_budget || !d_p) return KVGOV_EINVAL;
    long long grid = ((long long)n_prob + (kThreads / 32) - 1) / (kThreads / 32);
    const long long cap = (long long)kvgov_host::sm_count() * 32;
    if (grid > cap) grid = cap;
    origami_kernel<<<(unsigned)grid, kThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        d_values, d_off, n_prob, d_budget, d_p, d_lambda, d_utility, d_status);
    return kvgov_host::launch_status();
}
