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

// Random-slot writes, the operations of an insert: kind 0 claims the
// slot's first 16 bytes with a 128-bit compare-and-swap from zero, kind 1
// claims it and then writes the second 16 bytes with one store, kind 2
// reads the first 16 bytes first (as the insert's look does) and then claims
// and writes.  Run on a zeroed table, every operation finds its slot empty.
template <int KIND>
__global__ void __launch_bounds__(kGatherThreads) slot_ops_kernel(unsigned long long *__restrict__ table,
                                                                  unsigned long long mask, long long n_ops,
                                                                  unsigned long long seed, uint32_t *sink) {
    const long long i = blockIdx.x * (long long)kGatherThreads + threadIdx.x;
    if (i >= n_ops) return;
    unsigned long long *p = table + 4 * (mix64(seed + (unsigned long long)i) & mask);
    const unsigned long long v = (seed + (unsigned long long)i) | 1ull;
    unsigned long long seen = 0ull;
    if (KIND == 2) {
        unsigned long long s0, s1;
        asm volatile("ld.global.v2.u64 {%0, %1}, [%2];\n" : "=l"(s0), "=l"(s1) : "l"(p) : "memory");
        seen = s0 | s1;
    }
    unsigned long long o0 = 0ull, o1 = 0ull;
    if (seen == 0ull) {
        asm volatile("{\n\t.reg .b128 c, n, o;\n\t"
                     "mov.b128 c, {%2, %3};\n\t"
                     "mov.b128 n, {%4, %5};\n\t"
                     "atom.relaxed.gpu.global.cas.b128 o, [%6], c, n;\n\t"
                     "mov.b128 {%0, %1}, o;\n\t}"
                     : "=l"(o0), "=l"(o1)
                     : "l"(0ull), "l"(0ull), "l"(v), "l"(v), "l"(p)
                     : "memory");
        if (KIND >= 1 && (o0 | o1) == 0ull)
            asm volatile("st.relaxed.gpu.global.v2.u64 [%0], {%1, %2};\n" ::"l"(p + 2), "l"(v), "l"(v) : "memory");
    }
    if ((o0 ^ seen) == 0x9e3779b97f4a7c15ull) sink[0] = 1u;
}

}  // namespace

extern "C" int kvgov_peak_slot_ops(void *d_table, uint64_t n_slots, int kind, int64_t n_ops, uint64_t seed,
                                   uint32_t *d_sink, kvgov_stream_t stream) {
    if (!d_table || !d_sink || n_slots == 0 || (n_slots & (n_slots - 1)) != 0 || n_ops < 0 || kind < 0 ||
        kind > 2 || (reinterpret_cast<uintptr_t>(d_table) & 15u) != 0)
        return 1;
    if (n_ops == 0) return 0;
    const long long blocks = (n_ops + kGatherThreads - 1) / kGatherThreads;
    if (blocks > 0x7fffffffll) return 1;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    unsigned long long *t = static_cast<unsigned long long *>(d_table);
    switch (kind) {
    case 0: slot_ops_kernel<0><<<(unsigned)blocks, kGatherThreads, 0, s>>>(t, n_slots - 1, n_ops, seed, d_sink); break;
    case 1: slot_ops_kernel<1><<<(unsigned)blocks, kGatherThreads, 0, s>>>(t, n_slots - 1, n_ops, seed, d_sink); break;
    default: slot_ops_kernel<2><<<(unsigned)blocks, kGatherThreads, 0, s>>>(t, n_slots - 1, n_ops, seed, d_sink); break;
    }
    return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

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
