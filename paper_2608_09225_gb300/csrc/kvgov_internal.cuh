// kvgov_internal.cuh -- helpers shared by the libkvgov translation units.
#pragma once
#include <cuda_runtime.h>
#include <cstdint>

#include "../../include/kvgov.h"

namespace kvgov_dev {

__device__ __forceinline__ void raise_flag(uint32_t *status, uint32_t flag) {
    if (status) atomicOr(status, flag);
}

// 16-byte asynchronous global->shared copy (LDGSTS, L2 only).  src_bytes < 16
// reads only that many bytes and zero-fills the rest of the destination.
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gmem_src, int src_bytes) {
    const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(gmem_src), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }

template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

}  // namespace kvgov_dev

namespace kvgov_host {

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline bool pow2_capacity(uint64_t cap) { return cap >= KVGOV_MIN_CAPACITY && (cap & (cap - 1)) == 0; }

// The bound on every wait of the insert protocol (kvgov_set_spin_limit).
uint32_t spin_limit();

// Arrival-order serving helpers (kvgov_arrival.cu).
int arrival_owner_min_by_request(const int64_t *d_blk_off, int32_t n_req, uint32_t *d_slot_of,
                                 uint64_t *d_owner, uint64_t seq_base, cudaStream_t stream);
bool arrival_args_ok(uint64_t capacity, uint64_t seq_base);

// The chain hash of a small batch (kvgov_chain_split.cu): the largest batch
// it takes, and its launch (arguments already checked by the caller).
long long chain_split_max_req();
int launch_chain_split(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                       const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                       const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                       uint32_t *d_status, cudaStream_t stream);

// kvgov_probe_resume, arguments already in the library's types (kvgov_table.cu).
int probe_resume(const uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests, const int64_t *d_blk_off,
                 int32_t n_req, int32_t *d_prefix_blocks, uint32_t *d_status, kvgov_stream_t stream);

// kvgov_insert_uncached; with d_gen, every slot or side-store entry it claims
// gets generation `gen` (kvgov_table.cu).
int insert_uncached_gen(uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests, const int64_t *d_blk_off,
                        int32_t n_req, const int32_t *d_prefix_blocks, unsigned long long *d_n_new,
                        uint32_t *d_status, uint32_t *d_gen, uint32_t gen, kvgov_stream_t stream);

// kvgov_chain_hash_insert_prev without the probe's completion: d_prefix_lower
// receives, for every request, a lower bound of its cached prefix on the
// table after the insert (what the chain launch's own lookups found while
// the insert ran; 0 where the batch was too small for them), which
// probe_resume completes (kvgov_chain.cu).
int chain_insert_prev_lower(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                            const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                            const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                            uint8_t *d_slots, uint64_t capacity, const uint8_t *d_prev_digests,
                            const int64_t *d_prev_blk_off, int32_t prev_n_req, const int32_t *d_prev_prefix_blocks,
                            int32_t *d_prefix_lower, unsigned long long *d_n_new, uint32_t *d_status,
                            kvgov_stream_t stream);

inline int launch_status() {
    return cudaGetLastError() == cudaSuccess ? KVGOV_OK : KVGOV_ECUDA;
}

inline int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 152;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 152;
    return n;
}

}  // namespace kvgov_host
