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
#include <atomic>
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

// One problem solved by the 32 lanes of a warp (any number of tenants): its
// n values v[0..n) and budget K_in; p_i goes to pout[i], which may be v
// itself (each lane reads a value before it writes that place).  `bad`
// flags the problem as malformed already.
__device__ __forceinline__ void solve_warp_core(const float *v, float *pout, long long n, float K_in, bool bad,
                                                long long q, float *__restrict__ lambda_out,
                                                float *__restrict__ utility_out, uint32_t *status) {
    const int lane = threadIdx.x & 31;
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
    float K = K_in;
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
        pout[i] = pi;
        if (!isnan(x)) my_u = fmaxf(my_u, usable(x) ? fminf(x, lam) : x);
    }
    const float u = warp_max(my_u);
    if (lane == 0) {
        if (lambda_out) lambda_out[q] = lam;
        if (utility_out) utility_out[q] = n > 0 ? u : 0.0f;
        if (bad) raise_flag(status, KVGOV_F_BADINDEX);
    }
}

// Problem q, its values and probabilities in global memory.
__device__ __forceinline__ void solve_warp(const float *__restrict__ values, const int64_t *__restrict__ off,
                                           long long q, long long total, const float *__restrict__ budget,
                                           float *__restrict__ p, float *__restrict__ lambda_out,
                                           float *__restrict__ utility_out, uint32_t *status) {
    const long long b0 = off[q], b1 = off[q + 1];
    const bool bad = b0 < 0 || b1 < b0 || b1 > total;
    const long long n = bad ? 0 : b1 - b0;
    const long long at = bad ? 0 : b0;
    solve_warp_core(values + at, p + at, n, budget[q], bad, q, lambda_out, utility_out, status);
}

// Reciprocal with the SFU's one-instruction approximation (relative error
// below 2^-22: within the tolerance the parity tests derive, which allows a
// few units in the last place per term).
__device__ __forceinline__ float rcp_approx(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// Loads in flight per thread while a CTA stages its values (16: one round
// trip for a CTA of 50-tenant problems; 4 took 109 us, 8 105, 16 92 on 2^20
// such problems), and partial sums per solver pass (independent add chains).
constexpr int kInFlight = 16;
constexpr int kAcc = 2;
__device__ __forceinline__ float acc_total(const float part[kAcc]) {
    float t = 0.0f;
#pragma unroll
    for (int a = 0; a < kAcc; ++a) t += part[a];
    return t;
}

// sum += r and m += 1 when r < t, as one compare and two predicated adds
// (no select per slot whose result would wait in a register).
__device__ __forceinline__ void add_if_below(float &sum, int &m, float r, float t) {
    asm("{\n\t.reg .pred on;\n\t"
        "setp.lt.f32 on, %2, %3;\n\t"
        "@on add.f32 %0, %0, %2;\n\t"
        "@on add.s32 %1, %1, 1;\n\t}"
        : "+f"(sum), "+r"(m)
        : "f"(r), "f"(t));
}

// One problem solved by one thread, its n <= kMax values x[0..n) staged in
// shared memory and held in registers for the solve: one pass over shared
// memory in and one out, every Newton step on registers (from shared memory
// the steps' re-reads made the kernel bound by its load pipe).  Every value
// is usable (the caller checked the CTA's values as it staged them), so the
// tenants above the level are found by one compare each: each value is
// replaced by its reciprocal, the padding slots kMax - n by +infinity (never
// above the level), and a tenant is above the level when 1 / v_i is below
// 1 / lambda, taken once per step.  The first Newton step -- every tenant
// above the level -- is folded into that pass; p_i = 1 - lambda * (1 / v_i).
// Register tiers of 16, 32, 50 (the paper's 50-tenant problems, section
// 5.5) and 64 slots.  The adversary's payoff is lambda (some tenant is
// usable whenever n > 0).
// CHECK: the values were not checked; the solver returns false, writing
// nothing, when one is not usable (r = 1 / v not positive and finite: v <= 0,
// NaN, infinite, or above 2^126, whose reciprocal is not a normal number;
// the warp solver takes those).
template <int kMax, bool CHECK = false>
__device__ __forceinline__ bool solve_thread_reg(float *x, int n, float K_in, long long q,
                                                 float *__restrict__ lambda_out, float *__restrict__ utility_out,
                                                 uint32_t *status) {
    float r[kMax];
    float part[kAcc];                                  // kAcc partial sums: independent add chains
    float rmin = __int_as_float(0x7f800000);
#pragma unroll
    for (int a = 0; a < kAcc; ++a) part[a] = 0.0f;
#pragma unroll
    for (int i = 0; i < kMax; ++i) {
        r[i] = i < n ? rcp_approx(x[i]) : __int_as_float(0x7f800000);
        if (i < n) part[i % kAcc] += r[i];
        if (CHECK) rmin = fminf(rmin, r[i]);
    }
    const float sum_all = acc_total(part);
    // a NaN or +infinity reciprocal makes the sum NaN or infinite
    if (CHECK && !(rmin > 0.0f && sum_all <= 3.0e38f)) return false;
    float K = K_in;
    const bool bad = !(K >= 0.0f);
    if (!(K >= 0.0f)) K = 0.0f;
    if (K > (float)n) K = (float)n;
    float lam;
    if (n == 0 || K <= 0.0f) {
        lam = 0.0f;                                   // nothing to spend: p = 0, lambda = the largest value
        for (int i = 0; i < n; ++i) lam = fmaxf(lam, x[i]);
    } else if (K >= (float)n) {
        lam = 0.0f;                                   // every tenant audited
    } else {
        lam = ((float)n - K) / sum_all;
        int prev_m = n;
        // a tenant on the level adds nothing either way: the budget curve is
        // continuous there
        for (int step = 0; step <= n; ++step) {
            const float t = rcp_approx(lam);
            float ps[kAcc];
            int pm[kAcc];
#pragma unroll
            for (int a = 0; a < kAcc; ++a) { ps[a] = 0.0f; pm[a] = 0; }
#pragma unroll
            for (int i = 0; i < kMax; ++i) add_if_below(ps[i % kAcc], pm[i % kAcc], r[i], t);
            const float sum = acc_total(ps);
            int m = 0;
#pragma unroll
            for (int a = 0; a < kAcc; ++a) m += pm[a];
            const float next = ((float)m - K) / sum;
            if (m == prev_m) { lam = next; break; }
            lam = fmaxf(lam, next);
            prev_m = m;
        }
    }
#pragma unroll
    for (int i = 0; i < kMax; ++i)
        if (i < n) x[i] = fmaxf(0.0f, 1.0f - lam * r[i]);
    if (lambda_out) lambda_out[q] = lam;
    if (utility_out) utility_out[q] = n > 0 ? lam : 0.0f;
    if (bad) raise_flag(status, KVGOV_F_BADINDEX);
    return true;
}

// kCta consecutive problems per CTA.  When every one of them has at most
// kSmallN tenants and every value is usable, the values are staged in shared
// memory with coalesced (16-byte where aligned) loads, a thread solves each
// problem, and the probabilities leave the same way: a few dozen
// instructions per problem per warp instead of a warp's reductions per
// problem.  Otherwise -- larger problems, or a value that is not a positive
// finite number somewhere in the CTA's span -- the CTA's warps take its
// problems one at a time (solve_warp), which handles every case.
constexpr int kCta = 128;
constexpr int kSmallN = 64;

// At most 96 registers, so that 5 CTAs fit an SM (102 unbounded: 4).
__global__ void __launch_bounds__(kCta, 5) origami_kernel(const float *__restrict__ values,
                                                       const int64_t *__restrict__ off, int32_t n_prob,
                                                       const float *__restrict__ budget, float *__restrict__ p,
                                                       float *__restrict__ lambda_out,
                                                       float *__restrict__ utility_out, uint32_t *status,
                                                       bool vec4) {
    __shared__ __align__(16) float sv[kCta * kSmallN + 4];
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
        // the span [base0, base1) lands at sv[lead ..], lead = base0 mod 4, so
        // that its 16-byte-aligned middle moves as float4 (vec4: values and p
        // are 16-byte aligned; else every element on its own)
        const int lead = vec4 ? (int)(base0 & 3) : 0;
        const int span = (int)(base1 - base0);
        const long long a0 = base0 - lead;                       // 16-byte aligned when vec4
        const int n4 = vec4 ? (lead + span) >> 2 : 0;            // whole float4 from a0
        const int tail0 = n4 > 0 ? 4 * n4 : lead;                // the first element after them
        bool usable_all = true;
        const float4 *v4 = reinterpret_cast<const float4 *>(values + a0);
        float4 *s4 = reinterpret_cast<float4 *>(sv);
        // kInFlight loads in flight per thread before their values are used
        for (int i0 = threadIdx.x; i0 < n4; i0 += kInFlight * kCta) {
            float4 c[kInFlight];
#pragma unroll
            for (int u = 0; u < kInFlight; ++u)
                if (i0 + u * kCta < n4) c[u] = __ldcs(v4 + i0 + u * kCta);
#pragma unroll
            for (int u = 0; u < kInFlight; ++u) {
                const int i = i0 + u * kCta;
                if (i < n4) {
                    s4[i] = c[u];
                    const int e = 4 * i;                         // element index from a0
                    usable_all &= (e < lead || usable(c[u].x)) && (e + 1 < lead || usable(c[u].y)) &&
                                  (e + 2 < lead || usable(c[u].z)) && usable(c[u].w);
                }
            }
        }
        for (int e = tail0 + threadIdx.x; e < lead + span; e += kCta) {    // the tail
            const float c = values[a0 + e];
            sv[e] = c;
            usable_all &= usable(c);
        }
        if (__syncthreads_and(usable_all)) {
            if (q < q1) {
                float *x = sv + lead + (my0 - base0);
                const int n = (int)(my1 - my0);
                const float K = budget[q];
                if (n <= 16) solve_thread_reg<16>(x, n, K, q, lambda_out, utility_out, status);
                else if (n <= 32) solve_thread_reg<32>(x, n, K, q, lambda_out, utility_out, status);
                else if (n <= 50) solve_thread_reg<50>(x, n, K, q, lambda_out, utility_out, status);
                else solve_thread_reg<kSmallN>(x, n, K, q, lambda_out, utility_out, status);
            }
            __syncthreads();
            // out: the same split; the lead elements and the tail are the span's own
            float4 *p4 = reinterpret_cast<float4 *>(p + a0);
            for (int i = threadIdx.x; i < n4; i += kCta) {
                const float4 c = s4[i];
                if (4 * i >= lead) {
                    __stcs(p4 + i, c);
                } else {                                         // the first float4 holds elements before the span
                    if (4 * i + 1 >= lead) p[a0 + 4 * i + 1] = c.y;
                    if (4 * i + 2 >= lead) p[a0 + 4 * i + 2] = c.z;
                    p[a0 + 4 * i + 3] = c.w;
                }
            }
            for (int e = tail0 + threadIdx.x; e < lead + span; e += kCta) p[a0 + e] = sv[e];
            return;
        }
    }
    for (long long qq = q0 + threadIdx.x / 32; qq < q1; qq += kCta / 32)
        solve_warp(values, off, qq, total, budget, p, lambda_out, utility_out, status);
}

// ---------------------------------------------------------------------------
// Streaming layout, for values and p on 16-byte boundaries: every warp of a
// persistent grid (3 CTAs of 4 warps per SM) walks the batch's warp tiles
// (32 problems each) on its own, with two shared-memory buffers.  The copy
// engine brings the warp's tile t + W into one buffer -- one bulk copy of
// the tile's span, rounded out to 16-byte bounds, completing on the
// buffer's mbarrier -- while the warp solves tile t in the other, in place,
// and the probabilities leave by one bulk store.  No warp waits for a global
// load or store of values, nor for another warp (a CTA-wide barrier per
// tile left warps waiting for the CTA's slowest Newton solve: 1.46 barrier
// stalls per issue), and the copies of some tiles overlap the solves of
// others.  A lane solves its problem in registers (solve_thread_reg, values
// checked as it goes); a problem it cannot take (a value that is not usable,
// more than kSmallN tenants, malformed offsets) is solved after by the whole
// warp, in place in the buffer; a tile whose span does not fit a buffer is
// solved warp-wide from global memory.

constexpr int kTile = 32;                         // problems per warp tile
constexpr int kBuf = kTile * kSmallN + 8;         // floats per buffer: a tile's span rounded out to 16 bytes
constexpr int kStreamWarps = kCta / 32;
constexpr uint32_t kBulkWaitLimit = 1u << 24;     // polls of a buffer's mbarrier before KVGOV_F_TIMEOUT
constexpr size_t kStreamSmem = 2 * kStreamWarps * kBuf * sizeof(float);

__device__ __forceinline__ uint32_t smem_u32(const void *ptr) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(ptr));
}
__device__ __forceinline__ void mbar_init(unsigned long long *bar) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bar)) : "memory");
}
// one arrival (the issuing thread's) and the bytes the bulk copy will deliver
__device__ __forceinline__ void mbar_arrive_tx(unsigned long long *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_done(unsigned long long *bar, uint32_t parity) {
    uint32_t done;
    asm volatile("{\n\t.reg .pred p;\n\t"
                 "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
                 "selp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(done)
                 : "r"(smem_u32(bar)), "r"(parity)
                 : "memory");
    return done != 0;
}
// Wait for the phase of the given parity to complete, at most kBulkWaitLimit
// polls; false if it did not.
__device__ bool mbar_wait(unsigned long long *bar, uint32_t parity) {
    for (uint32_t i = 0; i < kBulkWaitLimit; ++i) {
        if (mbar_done(bar, parity)) return true;
        if (i >= 32) __nanosleep(64);
    }
    return false;
}
__device__ __forceinline__ void bulk_load(float *dst, const float *src, uint32_t bytes, unsigned long long *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ void bulk_store(float *dst, const float *src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_u32(src)),
                 "r"(bytes)
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// the issuing thread's bulk stores have read their shared-memory source
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// ... and are complete
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// this thread's shared-memory writes, ordered before the bulk copies that follow
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ long long round_down4(long long e) { return e & ~3ll; }
__device__ __forceinline__ long long round_up4(long long e) { return (e + 3) & ~3ll; }

__global__ void __launch_bounds__(kCta, 3) origami_stream_kernel(const float *__restrict__ values,
                                                              const int64_t *__restrict__ off, int32_t n_prob,
                                                              const float *__restrict__ budget,
                                                              float *__restrict__ p, float *__restrict__ lambda_out,
                                                              float *__restrict__ utility_out, uint32_t *status) {
    extern __shared__ __align__(16) float dyn[];
    __shared__ unsigned long long s_bar[kStreamWarps][2];
    __shared__ long long s_b0[kStreamWarps][2], s_b1[kStreamWarps][2];   // the span of the tile in each buffer
    __shared__ int s_fits[kStreamWarps][2];                              // ... and whether it fits the buffer

    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const long long total = off[n_prob];
    const long long n_tiles = ((long long)n_prob + kTile - 1) / kTile;
    const long long W = (long long)gridDim.x * kStreamWarps;            // warps in the grid
    const long long t_first = (long long)blockIdx.x * kStreamWarps + w;
    if (t_first >= n_tiles) return;               // this warp has no tile (no CTA-wide barrier follows)
    float *const bufs = dyn + w * 2 * kBuf;

    // Lane 0: the copy of tile t (span [b0, b1)) into buffer b.  Elements
    // from round_down4(b0) land at the buffer's start; at the array's end the
    // last < 4 values come by plain loads.
    auto issue = [&](int b, long long b0, long long b1) {
        const bool fits = b0 >= 0 && b1 >= b0 && b1 <= total && b1 - b0 <= (long long)kTile * kSmallN;
        float *buf = bufs + b * kBuf;
        uint32_t bytes = 0;
        long long a0 = 0, a1 = 0;
        if (fits) {
            a0 = round_down4(b0);
            a1 = round_up4(b1) <= total ? round_up4(b1) : round_down4(b1);
            if (a1 > a0) bytes = (uint32_t)(4 * (a1 - a0));
        }
        s_b0[w][b] = b0;
        s_b1[w][b] = b1;
        s_fits[w][b] = fits;
        mbar_arrive_tx(&s_bar[w][b], bytes);
        if (bytes) bulk_load(buf, values + a0, bytes, &s_bar[w][b]);
        if (fits)
            for (long long e = a1 > b0 ? a1 : b0; e < b1; ++e) buf[e - a0] = values[e];
    };
    // lane 0: tile t's span, read one tile ahead of its copy
    auto read_span = [&](long long t, long long &b0, long long &b1) {
        b0 = b1 = 0;
        if (t < n_tiles) {
            const long long q0 = t * kTile, q1 = q0 + kTile < n_prob ? q0 + kTile : (long long)n_prob;
            b0 = off[q0];
            b1 = off[q1];
        }
    };
    // tile t's problem for this lane, read one tile ahead
    auto read_mine = [&](long long t, long long &m0, long long &m1, float &K) {
        const long long q = t * kTile + lane;
        m0 = m1 = 0;
        K = 0.0f;
        if (t < n_tiles && q < n_prob) {
            m0 = off[q];
            m1 = off[q + 1];
            K = budget[q];
        }
    };

    long long nb0 = 0, nb1 = 0;                   // lane 0: the span of the tile to issue next
    if (lane == 0) {
        mbar_init(&s_bar[w][0]);
        mbar_init(&s_bar[w][1]);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");   // before the copies use them
        long long b0, b1;
        read_span(t_first, b0, b1);
        issue(0, b0, b1);
        read_span(t_first + W, nb0, nb1);
    }
    long long m0, m1;
    float K;
    read_mine(t_first, m0, m1, K);
    __syncwarp();

    uint32_t parity[2] = {0u, 0u};
    bool aborted = false;
    int b = 0;
    for (long long t = t_first; t < n_tiles; t += W, b ^= 1) {
        // the next tile into the other buffer, once its last store has read it
        if (lane == 0 && t + W < n_tiles) {
            bulk_wait_read();
            issue(b ^ 1, nb0, nb1);
            read_span(t + 2 * W, nb0, nb1);
        }
        const bool arrived = mbar_wait(&s_bar[w][b], parity[b]);
        if (__any_sync(0xffffffffu, !arrived)) {  // the copy never completed: stop (the tile's data is not there)
            if (lane == 0) raise_flag(status, KVGOV_F_TIMEOUT);
            aborted = true;
            break;
        }
        parity[b] ^= 1u;
        const long long b0 = s_b0[w][b], b1 = s_b1[w][b];
        const bool fits = s_fits[w][b] != 0;
        const long long q = t * kTile + lane;
        const long long q1 = t * kTile + kTile < n_prob ? t * kTile + kTile : (long long)n_prob;
        long long nm0, nm1;                       // this lane's problem of the next tile
        float nK;
        read_mine(t + W, nm0, nm1, nK);
        float *buf = bufs + b * kBuf;
        const long long a0 = round_down4(b0);
        if (fits) {
            bool left = false;                    // this lane's problem is left to the warp
            if (q < q1) {
                const bool ok = m0 >= b0 && m1 >= m0 && m1 <= b1 && m1 - m0 <= kSmallN;
                const int n = ok ? (int)(m1 - m0) : 0;
                float *x = buf + (m0 - a0);
                bool done = false;
                if (ok) {
                    if (n <= 16) done = solve_thread_reg<16, true>(x, n, K, q, lambda_out, utility_out, status);
                    else if (n <= 32) done = solve_thread_reg<32, true>(x, n, K, q, lambda_out, utility_out, status);
                    else if (n <= 50) done = solve_thread_reg<50, true>(x, n, K, q, lambda_out, utility_out, status);
                    else done = solve_thread_reg<kSmallN, true>(x, n, K, q, lambda_out, utility_out, status);
                }
                left = !done;
            }
            __syncwarp();
            for (unsigned pend = __ballot_sync(0xffffffffu, left); pend; pend &= pend - 1) {
                const long long dq = t * kTile + (__ffs((int)pend) - 1);
                const long long d0 = off[dq], d1 = off[dq + 1];
                if (d0 >= b0 && d1 >= d0 && d1 <= b1)
                    solve_warp_core(buf + (d0 - a0), buf + (d0 - a0), d1 - d0, budget[dq], false, dq, lambda_out,
                                    utility_out, status);
                else
                    solve_warp(values, off, dq, total, budget, p, lambda_out, utility_out, status);
                __syncwarp();
            }
            fence_async_smem();
            __syncwarp();
            if (lane == 0) {                      // [b0, b1) out: its 16-byte-aligned middle in one bulk store
                const long long c0 = round_up4(b0) < b1 ? round_up4(b0) : b1;
                const long long c1 = round_down4(b1) > c0 ? round_down4(b1) : c0;
                for (long long e = b0; e < c0; ++e) p[e] = buf[e - a0];
                for (long long e = c1; e < b1; ++e) p[e] = buf[e - a0];
                if (c1 > c0) bulk_store(p + c0, buf + (c0 - a0), (uint32_t)(4 * (c1 - c0)));
            }
        } else {
            for (long long qq = t * kTile; qq < q1; ++qq)
                solve_warp(values, off, qq, total, budget, p, lambda_out, utility_out, status);
        }
        __syncwarp();                             // buffer b's next copy may go once its store has read it
        m0 = nm0;
        m1 = nm1;
        K = nK;
    }
    if (lane == 0) {
        bulk_wait_all();
        if (aborted)                              // copies that may still be under way into either buffer
            for (int k = 0; k < 2; ++k) mbar_wait(&s_bar[w][k], parity[k]);
    }
}

// CTAs of origami_stream_kernel resident at once on the current device
// (its shared memory set up), looked up once per device; 0 if it cannot run.
int stream_ctas() {
    static std::atomic<int> cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    int v = cache[dev].load(std::memory_order_relaxed);
    if (v == 0) {
        int per_sm = 0, sms = 0;
        if (cudaFuncSetAttribute(origami_stream_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kStreamSmem) != cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, origami_stream_kernel, kCta, kStreamSmem) !=
                cudaSuccess ||
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
            cudaGetLastError();
            return 0;
        }
        v = per_sm > 0 ? per_sm * sms : -1;
        cache[dev].store(v, std::memory_order_relaxed);
    }
    return v > 0 ? v : 0;
}

}  // namespace

extern "C" int kvgov_origami(const float *d_values, const int64_t *d_off, int32_t n_prob, const float *d_budget,
                             float *d_p, float *d_lambda, float *d_utility, uint32_t *d_status,
                             kvgov_stream_t stream) {
    if (n_prob < 0 || !d_off) return KVGOV_EINVAL;
    if (n_prob == 0) return KVGOV_OK;
    if (!d_values || !d_budget || !d_p) return KVGOV_EINVAL;
    const long long grid = ((long long)n_prob + kCta - 1) / kCta;
    const bool vec4 = kvgov_host::aligned16(d_values) && kvgov_host::aligned16(d_p);
    const int resident = vec4 ? stream_ctas() : 0;
    if (resident > 0) {
        const long long ctas = ((long long)n_prob + kTile * kStreamWarps - 1) / (kTile * kStreamWarps);
        const long long g = ctas < resident ? ctas : resident;
        origami_stream_kernel<<<(unsigned)g, kCta, kStreamSmem, reinterpret_cast<cudaStream_t>(stream)>>>(
            d_values, d_off, n_prob, d_budget, d_p, d_lambda, d_utility, d_status);
    } else {
        origami_kernel<<<(unsigned)grid, kCta, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
            d_values, d_off, n_prob, d_budget, d_p, d_lambda, d_utility, d_status, vec4);
    }
    return kvgov_host::launch_status();
}
