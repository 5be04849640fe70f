// kvgov_origami.cu -- ORIGAMI audit allocation, batched (kvgov_origami).
//
// Paper: section 4.3, Theorem (ORIGAMI water-filling solution).  The defender
// spreads an audit budget K over tenants with values at risk v_i > 0 to
// minimise the adversary's best payoff max_i v_i (1 - p_i) subject to
// sum_i p_i = K, p_i in [0, 1]; the optimum is p_i = max(0, 1 - lambda / v_i)
// with the unique water level lambda meeting the budget.
//
// In fp32.  The budget as a function of the level,
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

// One problem solved by the 32 lanes of a warp (any number of tenants).
__device__ __forceinline__ void solve_warp(const float *__restrict__ values, const int64_t *__restrict__ off,
                                           long long q, long long total, const float *__restrict__ budget,
                                           float *__restrict__ p, float *__restrict__ lambda_out,
                                           float *__restrict__ utility_out, uint32_t *status) {
    const int lane = threadIdx.x & 31;
    const long long b0 = off[q], b1 = off[q + 1];
    bool bad = b0 < 0 || b1 < b0 || b1 > total;
    const long long n = bad ? 0 : b1 - b0;
    const float *v = values + (bad ? 0 : b0);

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
    } else {
        lam = 0.0f;
        int prev_m = -1;
        for (int step = 0; step <= npos + 1; ++step) {          // warp-uniform
            float sum = 0.0f;
            int m = 0;
            for (long long i = lane; i < n; i += 32) {
                const float x = v[i];
                if (usable(x) && x > lam) { sum += __frcp_rn(x); ++m; }
            }
            sum = warp_sum(sum);
            m = warp_isum(m);
            const float next = ((float)m - K) / sum;
            if (m == prev_m) { lam = next; break; }
            lam = fmaxf(lam, next);
            prev_m = m;
        }
    }

    // p_i, and the adversary's payoff v_i (1 - p_i): min(v_i, lambda) for a
    // usable tenant (lambda where audited, v_i where not), written that way
    // because 1 - p_i cancels when p_i is close to 1.
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

// Reciprocal with the SFU's one-instruction approximation (relative error
// below 2^-22: within the tolerance the parity tests derive, which allows a
// few units in the last place per term).
__device__ __forceinline__ float rcp_approx(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// One problem solved by one thread, its n <= kMax values x[0..n) staged in
// shared memory and held in registers for the solve: one pass over shared
// memory in and one out, every Newton step on registers (from shared memory
// the steps' re-reads made the kernel bound by its load pipe).  Each value
// is replaced by its reciprocal (+infinity for a tenant that is not usable,
// which then never counts as above the level and gets p = 0): the steps
// compare lambda * (1 / v_i) with 1 and sum reciprocals, with no division
// per tenant, and p_i = 1 - lambda * (1 / v_i).  The kMax - n padding slots
// hold 0 -- not usable, not flagged, adding exactly 0 to every sum.  Register
// tiers of 16, 32, 50 (the paper's 50-tenant problems, section 5.5) and 64
// slots.  The
// adversary's payoff is lambda whenever a tenant is usable (min(v_i, lambda)
// over the usable ones, the others at most 0), else the largest value.
template <int kMax>
__device__ __forceinline__ void solve_thread_reg(float *x, const float *__restrict__ vg, int n, float K_in,
                                                 long long q, float *__restrict__ lambda_out,
                                                 float *__restrict__ utility_out, uint32_t *status) {
    float r[kMax];
    int npos = 0, nbad = 0;
    float vmax = 0.0f, sum_all = 0.0f;
#pragma unroll
    for (int i = 0; i < kMax; ++i) {
        const float xi = i < n ? x[i] : 0.0f;
        const bool use = usable(xi);
        npos += use;
        nbad += !use && !(xi <= 0.0f);
        vmax = use ? fmaxf(vmax, xi) : vmax;
        r[i] = use ? rcp_approx(xi) : __int_as_float(0x7f800000);
        sum_all += use ? r[i] : 0.0f;
    }
    float K = K_in;
    const bool bad = nbad > 0 || !(K >= 0.0f);
    if (!(K >= 0.0f)) K = 0.0f;
    if (K > (float)npos) K = (float)npos;
    float lam;
    if (npos == 0 || K <= 0.0f) {
        lam = vmax;
    } else if (K >= (float)npos) {
        lam = 0.0f;
    } else {
        lam = ((float)npos - K) / sum_all;
        int prev_m = npos;
        // a tenant is above the level when 1 / v_i is below 1 / lambda: one
        // compare per tenant against a threshold taken once per step (a tenant
        // on the level adds nothing either way: the budget curve is continuous
        // there)
        for (int step = 0; step <= npos; ++step) {
            const float t = rcp_approx(lam);
            float sum = 0.0f;
            int m = 0;
#pragma unroll
            for (int i = 0; i < kMax; ++i) {
                const bool on = r[i] < t;
                sum += on ? r[i] : 0.0f;
                m += on;
            }
            const float next = ((float)m - K) / sum;
            if (m == prev_m) { lam = next; break; }
            lam = fmaxf(lam, next);
            prev_m = m;
        }
    }
#pragma unroll
    for (int i = 0; i < kMax; ++i)
        if (i < n) x[i] = fmaxf(0.0f, 1.0f - lam * r[i]);
    float u = lam;
    if (npos == 0) {
        u = n > 0 ? -3.0e38f : 0.0f;
        for (int i = 0; i < n; ++i) {
            const float xi = vg[i];
            if (!isnan(xi)) u = fmaxf(u, xi);
        }
    }
    if (lambda_out) lambda_out[q] = lam;
    if (utility_out) utility_out[q] = u;
    if (bad) raise_flag(status, KVGOV_F_BADINDEX);
}

// kCta consecutive problems per CTA.  When every one of them has at most
// kSmallN tenants, their values are staged in shared memory with coalesced
// loads, a thread solves each problem, and the probabilities leave with
// coalesced stores: a few dozen instructions per problem per warp instead
// of a warp's reductions per problem.  Otherwise the CTA's warps take its
// problems one at a time (solve_warp).
constexpr int kCta = 128;
constexpr int kSmallN = 64;

__global__ void __launch_bounds__(kCta) origami_kernel(const float *__restrict__ values,
                                                       const int64_t *__restrict__ off, int32_t n_prob,
                                                       const float *__restrict__ budget, float *__restrict__ p,
                                                       float *__restrict__ lambda_out,
                                                       float *__restrict__ utility_out, uint32_t *status) {
    __shared__ float sv[kCta * kSmallN];
    const long long total = off[n_prob];
    const long long q0 = (long long)blockIdx.x * kCta;
    const long long q1 = q0 + kCta < n_prob ? q0 + kCta : (long long)n_prob;
    const long long q = q0 + threadIdx.x;
    const long long base0 = off[q0], base1 = off[q1];
    long long my0 = 0, my1 = 0;
    bool ok = true;
    if (q < q1) {
        my0 = off[q];
        my1 = off[q + 1];
        ok = my0 >= base0 && my1 >= my0 && my1 <= base1 && my1 - my0 <= kSmallN;
    }
    ok = ok && base0 >= 0 && base1 >= base0 && base1 <= total && base1 - base0 <= kCta * kSmallN;
    if (__syncthreads_and(ok)) {
        const int span = (int)(base1 - base0);
        for (int i = threadIdx.x; i < span; i += kCta) sv[i] = values[base0 + i];
        __syncthreads();
        if (q < q1) {
            float *x = sv + (my0 - base0);
            const int n = (int)(my1 - my0);
            if (n <= 16) solve_thread_reg<16>(x, values + my0, n, budget[q], q, lambda_out, utility_out, status);
            else if (n <= 32) solve_thread_reg<32>(x, values + my0, n, budget[q], q, lambda_out, utility_out, status);
            else if (n <= 50) solve_thread_reg<50>(x, values + my0, n, budget[q], q, lambda_out, utility_out, status);
            else solve_thread_reg<kSmallN>(x, values + my0, n, budget[q], q, lambda_out, utility_out, status);
        }
        __syncthreads();
        for (int i = threadIdx.x; i < span; i += kCta) p[base0 + i] = sv[i];
    } else {
        for (long long qq = q0 + threadIdx.x / 32; qq < q1; qq += kCta / 32)
            solve_warp(values, off, qq, total, budget, p, lambda_out, utility_out, status);
    }
}

}  // namespace

extern "C" int kvgov_origami(const float *d_values, const int64_t *d_off, int32_t n_prob, const float *d_budget,
                             float *d_p, float *d_lambda, float *d_utility, uint32_t *d_status,
                             kvgov_stream_t stream) {
    if (n_prob < 0 || !d_off) return KVGOV_EINVAL;
    if (n_prob == 0) return KVGOV_OK;
    if (!d_values || !d_budget || !d_p) return KVGOV_EINVAL;
    const long long grid = ((long long)n_prob + kCta - 1) / kCta;
    origami_kernel<<<(unsigned)grid, kCta, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        d_values, d_off, n_prob, d_budget, d_p, d_lambda, d_utility, d_status);
    return kvgov_host::launch_status();
}
