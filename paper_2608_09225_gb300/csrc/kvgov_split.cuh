// kvgov_split.cuh -- pieces shared by the two-warp kernels of libkvgov
// (kvgov_chain_split.cu, kvgov_response.cu): a round warp runs SHA-256
// rounds with K_t + W_t read from shared memory, a schedule warp on another
// SM sub-partition builds the messages and expands their schedules
// (FIPS 180-4 section 6.2.2 step 1) into that memory, and the two meet on
// named barriers of 64 threads.  K_t + W_t are stored as uint4 [t / 4][lane],
// so that the round warp reads four rounds' values with one 16-byte load.
#pragma once
#include <cstdint>

#include "sha256_dev.cuh"

namespace kvgov_dev {

// Named barriers of the pair's 64 threads.  Each is executed by a whole warp
// at once (the lanes are reconverged first: some code before them is
// per-lane).
__device__ __forceinline__ void bar_sync(int id) {
    __syncwarp();
    asm volatile("bar.sync %0, 64;\n" ::"r"(id) : "memory");
}
__device__ __forceinline__ void bar_arrive(int id) {
    __syncwarp();
    asm volatile("bar.arrive %0, 64;\n" ::"r"(id) : "memory");
}

__device__ __forceinline__ void load16(const uint4 (*kw)[32], int lane, uint32_t k[16]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint4 x = kw[i][lane];
        k[4 * i] = x.x; k[4 * i + 1] = x.y; k[4 * i + 2] = x.z; k[4 * i + 3] = x.w;
    }
}

// K_t + W_t, t = 0..15, of a message w into kw[0..3].
__device__ __forceinline__ void store_kw16(const uint32_t w[16], uint4 (*kw)[32], int lane) {
#pragma unroll
    for (int i = 0; i < 4; ++i)
        kw[i][lane] = make_uint4(w[4 * i] + sha_k(4 * i), w[4 * i + 1] + sha_k(4 * i + 1),
                                 w[4 * i + 2] + sha_k(4 * i + 2), w[4 * i + 3] + sha_k(4 * i + 3));
}

// One chunk of the message schedule (FIPS 180-4 section 6.2.2 step 1): w
// holds W_{16(q-1)} .. W_{16q-1} and becomes W_{16q} .. W_{16q+15}.
__device__ __forceinline__ void schedule_chunk(uint32_t w[16]) {
#pragma unroll
    for (int t = 0; t < 16; ++t)
        w[t] = w[t] + w[(t + 9) & 15] + ssig0(w[(t + 1) & 15]) + ssig1(w[(t + 14) & 15]);
}

// K_t + W_t of chunk q (w = W_{16q} .. W_{16q+15}) into kw[4 (q - 1) ..].
__device__ __forceinline__ void store_kw_chunk(const uint32_t w[16], uint4 (*kw)[32], int lane, int q) {
#pragma unroll
    for (int i = 0; i < 4; ++i)
        kw[4 * (q - 1) + i][lane] =
            make_uint4(w[4 * i] + c_sha_k[16 * q + 4 * i], w[4 * i + 1] + c_sha_k[16 * q + 4 * i + 1],
                       w[4 * i + 2] + c_sha_k[16 * q + 4 * i + 2], w[4 * i + 3] + c_sha_k[16 * q + 4 * i + 3]);
}

// The schedule warp's half of a compression: expand the message w[0..15]
// (FIPS 180-4 section 6.2.2 step 1) into K_t + W_t for t = 16..63, chunk q
// = t / 16 stored to kw[4 (q - 1) ..]; bar0 >= 0: arrive on barrier
// bar0 + q - 1 after chunk q.  w is overwritten.
__device__ __forceinline__ void schedule_kw48(uint32_t w[16], uint4 (*kw)[32], int lane, int bar0) {
#pragma unroll 1
    for (int q = 1; q < 4; ++q) {
        schedule_chunk(w);
        store_kw_chunk(w, kw, lane, q);
        if (bar0 >= 0) bar_arrive(bar0 + q - 1);
    }
}

}  // namespace kvgov_dev
