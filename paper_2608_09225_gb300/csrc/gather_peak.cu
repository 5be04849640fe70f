// gather_peak.cu -- random-slot read microbenchmark (libkvgov_peak.so; header
// include/kvgov_peak.h): the bandwidth ceiling of the table kernels.
//
// A probe or insert reads 16 or 32 bytes at a pseudo-random slot of a table
// far larger than L2, so it cannot reach the streaming copy bandwidth: every
// 32-byte read pulls a whole DRAM burst.  This kernel issues nothing but such
// reads (8 independent ones per thread, slot = mix64(seed + read index) &
// mask) and folds the loaded words into a value that is written only in a
// case that never happens, so the loads stay live.
#include <cuda_runtime.h>
#include <cstdint>

#include "../../include/kvgov_peak.h"

namespace {

constexpr int kGatherThreads = 256;
constexpr int kReadsPerThread = 8;

// The splitmix64 output function (Steele, Lea and Flood, 2014): a bijective
// 64-bit mixer, so consecutive read indices land on unrelated slots.
__device__ __forceinline__ unsigned long long mix64(unsigned long long z) {
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
    return z ^ (z >> 31);
}

template <bool WHOLE_SLOT>
__global__ void __launch_bounds__(kGatherThreads) gather_kernel(const uint4 *__restrict__ table,
                                                                unsigned long long mask, long long n_reads,
                                                                unsigned long long seed, uint32_t *sink) {
    const long long base = (blockIdx.x * (long long)kGatherThreads + threadIdx.x) * kReadsPerThread;
    uint32_t acc = 0;
#pragma unroll
    for (int k = 0; k < kReadsPerThread; ++k) {
        if (base + k < n_reads) {
            const unsigned long long slot = mix64(seed + (unsigned long long)(base + k)) & mask;
            const uint4 a = __ldg(table + 2 * slot);
            acc ^= a.x ^ a.y ^ a.z ^ a.w;
            if (WHOLE_SLOT) {
                const uint4 b = __ldg(table + 2 * slot + 1);
                acc ^= b.x ^ b.y ^ b.z ^ b.w;
            }
        }
    }
    if (acc == 0x9e3779b9u) sink[0] = acc;
}

}  // namespace

extern "C" int kvgov_peak_gather(const void *d_table, uint64_t n_slots, int slot_bytes, int64_t n_reads,
                                 uint64_t seed, uint32_t *d_sink, kvgov_stream_t stream) {
    if (!d_table || !d_sink || n_slots == 0 || (n_slots & (n_slots - 1)) != 0 || n_reads < 0 ||
        (slot_bytes != 16 && slot_bytes != 32) || (reinterpret_cast<uintptr_t>(d_table) & 15u) != 0)
        return 1;
    if (n_reads == 0) return 0;
    const long long per_cta = (long long)kGatherThreads * kReadsPerThread;
    const long long blocks = (n_reads + per_cta - 1) / per_cta;
    if (blocks > 0x7fffffffll) return 1;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const uint4 *t = static_cast<const uint4 *>(d_table);
    if (slot_bytes == 32)
        gather_kernel<true><<<(unsigned)blocks, kGatherThreads, 0, s>>>(t, n_slots - 1, n_reads, seed, d_sink);
    else
        gather_kernel<false><<<(unsigned)blocks, kGatherThreads, 0, s>>>(t, n_slots - 1, n_reads, seed, d_sink);
    return cudaGetLastError() == cudaSuccess ? 0 : 2;
}
