// kvgov_salts.cu -- per-principal salts, paper section 4.1:
// sigma_p = HMAC_K(secret, principal_id), with HMAC as RFC 2104 defines it
// over SHA-256 (block 64 bytes, output 32 bytes):
//   K0 = secret zero-padded to 64 bytes (SHA-256(secret) first if longer),
//   sigma_p = H((K0 ^ opad) || H((K0 ^ ipad) || id_p)).
//
// The secret travels in the launch parameters.  Each CTA absorbs K0^ipad and
// K0^opad once (two compressions, plus the key hash for long keys) into
// shared memory; each thread then finishes one principal's inner hash over
// its id bytes and the single-block outer hash.
#include "kvgov_internal.cuh"
#include "sha256_dev.cuh"

namespace {

using namespace kvgov_dev;

constexpr int kSaltThreads = 64;

struct SaltParams {
    uint8_t secret[KVGOV_MAX_SECRET];
    const uint8_t *ids;
    const int64_t *id_off;
    uint8_t *salts;
    uint32_t *status;
    uint32_t secret_len;
    int32_t n;
};

// Continue SHA-256 from state s, which has absorbed `prior` bytes (a multiple
// of 64), over len more bytes get(0..len-1), then pad (FIPS 180-4 section
// 5.1.1) for the total length and finish.
template <class Get>
__device__ void sha_absorb_finish(uint32_t s[8], unsigned long long prior, unsigned long long len, Get get) {
    const unsigned long long total_bits = (prior + len) * 8ull;
    const unsigned long long padded = ((len + 9ull + 63ull) / 64ull) * 64ull;
    for (unsigned long long off = 0; off < padded; off += 64) {
        uint32_t w[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            uint32_t v = 0;
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                const unsigned long long idx = off + 4ull * i + b;
                const uint32_t byte = idx < len ? (uint32_t)get(idx) : (idx == len ? 0x80u : 0u);
                v = (v << 8) | byte;
            }
            w[i] = v;
        }
        if (off + 64 == padded) {
            w[14] = (uint32_t)(total_bits >> 32);
            w[15] = (uint32_t)total_bits;
        }
        sha_compress_small(s, w);
    }
}

// K0 of RFC 2104 as 16 big-endian words: the key zero-padded to 64 bytes, or
// SHA-256(key) zero-padded when the key is longer than 64 bytes.
__device__ __forceinline__ void hmac_k0(const SaltParams &p, uint32_t k0[16]) {
    if (p.secret_len > 64) {
        uint32_t hk[8];
        sha_iv(hk);
        sha_absorb_finish(hk, 0ull, p.secret_len, [&](unsigned long long i) { return p.secret[i]; });
#pragma unroll
        for (int i = 0; i < 16; ++i) k0[i] = i < 8 ? hk[i] : 0u;
        return;
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        uint32_t v = 0;
#pragma unroll
        for (int b = 0; b < 4; ++b) v = (v << 8) | (4u * i + b < p.secret_len ? (uint32_t)p.secret[4 * i + b] : 0u);
        k0[i] = v;
    }
}

__global__ void __launch_bounds__(kSaltThreads) salts_kernel(const SaltParams p) {
    // The (K0 ^ ipad) and (K0 ^ opad) midstates are computed once per CTA,
    // by the first thread of warp 0 and of warp 1 in parallel.
    __shared__ uint32_t s_mid[2][8];
    if ((threadIdx.x & 31) == 0 && threadIdx.x < 64) {
        const uint32_t pad = threadIdx.x == 0 ? 0x36363636u : 0x5c5c5c5cu;
        uint32_t k0[16], st[8];
        hmac_k0(p, k0);
#pragma unroll
        for (int i = 0; i < 16; ++i) k0[i] ^= pad;
        sha_iv(st);
        sha_compress_small(st, k0);
#pragma unroll
        for (int i = 0; i < 8; ++i) s_mid[threadIdx.x >> 5][i] = st[i];
    }
    __syncthreads();
    uint32_t *s_ipad = s_mid[0], *s_opad = s_mid[1];

    for (long long pr = (long long)blockIdx.x * kSaltThreads + threadIdx.x; pr < p.n;
         pr += (long long)gridDim.x * kSaltThreads) {
        const long long a = p.id_off[pr], b = p.id_off[pr + 1];
        if (a < 0 || b < a) {
            raise_flag(p.status, KVGOV_F_BADINDEX);
            continue;
        }
        const uint8_t *id = p.ids + a;
        uint32_t inner[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) inner[i] = s_ipad[i];
        sha_absorb_finish(inner, 64ull, (unsigned long long)(b - a), [&](unsigned long long i) { return id[i]; });

        // outer: (K0 ^ opad) already absorbed; one block = inner digest + padding
        uint32_t s[8], w[16];
#pragma unroll
        for (int i = 0; i < 8; ++i) { s[i] = s_opad[i]; w[i] = inner[i]; }
        w[8] = 0x80000000u;
#pragma unroll
        for (int i = 9; i < 15; ++i) w[i] = 0u;
        w[15] = (64u + 32u) * 8u;
        sha_compress_small(s, w);

        uint4 *dst = reinterpret_cast<uint4 *>(p.salts + 32ll * pr);
        dst[0] = make_uint4(bswap32(s[0]), bswap32(s[1]), bswap32(s[2]), bswap32(s[3]));
        dst[1] = make_uint4(bswap32(s[4]), bswap32(s[5]), bswap32(s[6]), bswap32(s[7]));
    }
}

}  // namespace

extern "C" int kvgov_derive_salts(const uint8_t *secret, size_t secret_len, const uint8_t *d_ids,
                                  const int64_t *d_id_off, int32_t n_principals, uint8_t *d_salts,
                                  uint32_t *d_status, kvgov_stream_t stream) {
    if (secret_len > KVGOV_MAX_SECRET || (secret_len > 0 && !secret)) return KVGOV_EINVAL;
    if (n_principals < 0) return KVGOV_EINVAL;
    if (!d_ids || !d_id_off || !d_salts || !kvgov_host::aligned16(d_salts)) return KVGOV_EINVAL;
    if (n_principals == 0) return KVGOV_OK;
    SaltParams p;
    for (size_t i = 0; i < KVGOV_MAX_SECRET; ++i) p.secret[i] = i < secret_len ? secret[i] : 0;
    p.ids = d_ids; p.id_off = d_id_off; p.salts = d_salts; p.status = d_status;
    p.secret_len = (uint32_t)secret_len; p.n = n_principals;
    long long grid = ((long long)n_principals + kSaltThreads - 1) / kSaltThreads;
    if (grid > 4096) grid = 4096;
    salts_kernel<<<(unsigned)grid, kSaltThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(p);
    return kvgov_host::launch_status();
}
