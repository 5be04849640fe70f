// int_peak.cu -- integer issue-rate microbenchmark for the roofline of the
// hashing kernels (libkvgov_peak.so; header include/kvgov_peak.h).
//
// Every thread runs `iters` iterations of a fixed body of integer
// instructions over register-resident values (no memory traffic).  Each CTA
// records its SM id and clock64() at start and end; the host divides the
// thread-operations an SM executed by the SM clock cycles it took, which
// gives thread-ops per SM clock, independent of the clock frequency.
//
// Kinds (ops per thread per iteration in kvgov_peak_ops_per_iter):
//   0  LOP3   x_s = lop3(x_s, x_{s+1}, x_{s+2})    over 8 streams
//   1  SHF    x_s = shf.r.wrap(x_s, x_{s+1}, n_s)   over 8 streams
//   2  IADD3  x_s = x_s + x_{s+1} + x_{s+2}         over 8 streams
//   3  SHA-256: one FIPS 180-4 compression (1384 nominal ops: 64 rounds x 14
//      + 48 schedule words x 10 + 8) on each of 2 independent chains, adds on
//      the ALU pipe
//   4  the same with every add issued as IMAD on the FMA pipe
//   5  IMAD  x_s = x_s * one + x_{s+1}   (one = 1 at run time)
//   6  SHA-256 rounds only (64 a iteration, K_t + W_t from registers, as the
//      small-batch chain kernel's round warp runs them): sha_rounds16_t1t2
//   7  the same with sha_rounds16_short
//   8  LOP3 on streams 0-3 and IADD3 on streams 4-7, interleaved
//   9  LOP3 on streams 0-3 and IMAD on streams 4-7
//  10  SHF on streams 0-3 and IADD3 on streams 4-7
//  11  the chain kernel's steady block: H(P || T), a 96-byte message = two
//      compact compressions (2 x 1384 nominal ops) on each of 2 independent
//      chains, every add on the ALU (sha_compress_small)
//  12  the same with the adds off the rounds' dependency chain on the FMA
//      pipe (sha_compress_small_split)
// Kinds 8-10 show whether two kinds of instruction share one pipe: if they
// do, the mix runs at the slower kind's rate; if not, it can run above it.
// Kinds 6 and 7 count 14 nominal ops a round; launched with one warp per SM
// sub-partition they give a lone warp's round rate.
// Each update reads two other streams' latest values, so no chain of updates
// collapses into fewer instructions (a three-input boolean of three fixed
// inputs would fold into one LOP3; these never have three fixed inputs).
#include <cuda_runtime.h>
#include <cstdint>

#include "../../include/kvgov_peak.h"
#include "sha256_dev.cuh"

namespace {

constexpr int kStreams = 8;
constexpr int kShaChains = 2;

__device__ __forceinline__ uint32_t smid() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
    return r;
}

template <int KIND>
__global__ void peak_kernel(int iters, uint32_t seed, uint32_t one, uint32_t *sink, unsigned long long *clocks) {
    __shared__ unsigned long long t_start;
    uint32_t x[kStreams];
#pragma unroll
    for (int s = 0; s < kStreams; ++s) x[s] = (seed ^ (threadIdx.x * 0x9e3779b9u)) + 0x85ebca6bu * (s + 1);
    __syncthreads();
    if (threadIdx.x == 0) t_start = clock64();
    __syncthreads();
    if (KIND == 6 || KIND == 7) {
        uint32_t v[8], kw[16];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = x[i];
#pragma unroll
        for (int i = 0; i < 16; ++i) kw[i] = x[i & 7] * (2u * i + 1u);
        for (int it = 0; it < iters; ++it) {
#pragma unroll 1
            for (int q = 0; q < 4; ++q) {
                if (KIND == 6) kvgov_dev::sha_rounds16_t1t2(v, kw);
                else kvgov_dev::sha_rounds16_short(v, kw);
            }
            kw[it & 15] ^= v[0];   // a new schedule word each iteration (one op per 64 rounds)
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) x[i] = v[i];
    } else if (KIND == 11 || KIND == 12) {
        uint32_t st[kShaChains][8];
#pragma unroll
        for (int c = 0; c < kShaChains; ++c) {
#pragma unroll
            for (int i = 0; i < 8; ++i) st[c][i] = x[i] + c;
        }
        for (int it = 0; it < iters; ++it) {
#pragma unroll
            for (int c = 0; c < kShaChains; ++c) {
                // H(st || T) with T = 16 words derived from st: two compressions from the IV
                uint32_t s[8], w[16];
                kvgov_dev::sha_iv(s);
#pragma unroll
                for (int i = 0; i < 8; ++i) { w[i] = st[c][i]; w[8 + i] = st[c][i] ^ (uint32_t)(it + i); }
                if (KIND == 11) kvgov_dev::sha_compress_small(s, w, kvgov_dev::AddAlu{});
                else kvgov_dev::sha_compress_small_split(s, w, kvgov_dev::AddFma{one});
#pragma unroll
                for (int i = 0; i < 8; ++i) w[i] = st[c][i] + (uint32_t)i;
                w[8] = 0x80000000u;
#pragma unroll
                for (int i = 9; i < 15; ++i) w[i] = 0u;
                w[15] = 96u * 8u;
                if (KIND == 11) kvgov_dev::sha_compress_small(s, w, kvgov_dev::AddAlu{});
                else kvgov_dev::sha_compress_small_split(s, w, kvgov_dev::AddFma{one});
#pragma unroll
                for (int i = 0; i < 8; ++i) st[c][i] = s[i];
            }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) x[i] = st[0][i] ^ st[1][i];
    } else if (KIND == 3 || KIND == 4) {
        uint32_t st[kShaChains][8], w[kShaChains][16];
#pragma unroll
        for (int c = 0; c < kShaChains; ++c) {
#pragma unroll
            for (int i = 0; i < 8; ++i) st[c][i] = x[i] + c;
        }
        for (int it = 0; it < iters; ++it) {
#pragma unroll
            for (int c = 0; c < kShaChains; ++c) {
#pragma unroll
                for (int i = 0; i < 16; ++i) w[c][i] = st[c][i & 7] ^ (uint32_t)i;
                if (KIND == 3) kvgov_dev::sha_compress(st[c], w[c], kvgov_dev::AddAlu{});
                else kvgov_dev::sha_compress(st[c], w[c], kvgov_dev::AddFma{one});
            }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) x[i] = st[0][i] ^ st[1][i];
    } else {
        for (int it = 0; it < iters; ++it) {
#pragma unroll
            for (int rep = 0; rep < 4; ++rep) {
#pragma unroll
                for (int s = 0; s < kStreams; ++s) {
                    const uint32_t a = x[(s + 1) % kStreams], b = x[(s + 2) % kStreams];
                    // the kind of instruction for this stream
                    const int op = KIND <= 2 || KIND == 5 ? KIND
                                 : (s < kStreams / 2 ? (KIND == 10 ? 1 : 0) : (KIND == 9 ? 5 : 2));
                    if (op == 0)
                        asm("lop3.b32 %0, %0, %1, %2, 0x96;" : "+r"(x[s]) : "r"(a), "r"(b));
                    else if (op == 1)
                        x[s] = __funnelshift_r(x[s], a, (s * 5 + rep * 3 + 1) & 31);
                    else if (op == 2)
                        x[s] = x[s] + a + b;
                    else
                        asm("mad.lo.u32 %0, %0, %1, %2;" : "+r"(x[s]) : "r"(one), "r"(a));
                }
            }
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const unsigned long long t_end = clock64();
        clocks[3 * blockIdx.x + 0] = smid();
        clocks[3 * blockIdx.x + 1] = t_start;
        clocks[3 * blockIdx.x + 2] = t_end;
    }
    uint32_t acc = 0;
#pragma unroll
    for (int s = 0; s < kStreams; ++s) acc ^= x[s];
    if (acc == 0x12345678u) sink[0] = acc;   // keeps every stream live
}

}  // namespace

extern "C" int kvgov_peak_ops_per_iter(int kind) {
    switch (kind) {
    case 0: case 1: return 4 * kStreams;   // one instruction per update; IADD3 counts as one op
    case 2: return 4 * kStreams;
    case 3: case 4: return kShaChains * 1384;
    case 5: return 4 * kStreams;
    case 6: case 7: return 64 * 14;
    case 8: case 9: case 10: return 4 * kStreams;
    case 11: case 12: return kShaChains * 2 * 1384;
    default: return 0;
    }
}

extern "C" int kvgov_peak_int(int kind, int iters, int blocks, int threads, uint32_t *d_sink,
                              unsigned long long *d_clocks, kvgov_stream_t stream) {
    if (kind < 0 || kind > 12 || iters <= 0 || blocks <= 0 || threads <= 0 || threads > 1024 || !d_sink ||
        !d_clocks)
        return 1;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    switch (kind) {
    case 0: peak_kernel<0><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 1: peak_kernel<1><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 2: peak_kernel<2><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 3: peak_kernel<3><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 4: peak_kernel<4><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 5: peak_kernel<5><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 6: peak_kernel<6><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 7: peak_kernel<7><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 8: peak_kernel<8><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 9: peak_kernel<9><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 10: peak_kernel<10><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    case 11: peak_kernel<11><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    default: peak_kernel<12><<<blocks, threads, 0, s>>>(iters, 1u, 1u, d_sink, d_clocks); break;
    }
    return cudaGetLastError() == cudaSuccess ? 0 : 2;
}
