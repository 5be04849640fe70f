// sha256_dev.cuh -- register-resident SHA-256 compression for sm_103a.
//
// SHA-256 as FIPS 180-4 defines it (section 4.1.2 functions, section 4.2.2
// constants, section 6.2.2 compression).  The paper fixes H = SHA-256 for
// block keys and for the HMAC salt (section 4.1; Table 9).
//
// Mapping onto the SM's integer pipes:
//   * every rotate is one funnel shift (SHF.R.W) via __funnelshift_r;
//   * the three-input boolean functions -- Ch, Maj and the XOR that closes
//     each Sigma / sigma -- are single LOP3 instructions, written as inline
//     PTX lop3.b32 with the truth table of the function;
//   * the 16-word message schedule is a rolling window in registers; with the
//     rounds fully unrolled every index is a compile-time constant, and the
//     round constants are immediates, so blocks whose schedule is known at
//     compile time (the final padding block of a fixed-length message) fold
//     to constants.
#pragma once
#include <cstdint>

namespace kvgov_dev {

// FIPS 180-4 section 4.2.2: K_0 .. K_63.  Returned through a switch so that,
// after unrolling, each use is an immediate operand.
__device__ __forceinline__ uint32_t sha_k(int t) {
    switch (t) {
    case 0: return 0x428a2f98u; case 1: return 0x71374491u; case 2: return 0xb5c0fbcfu; case 3: return 0xe9b5dba5u;
    case 4: return 0x3956c25bu; case 5: return 0x59f111f1u; case 6: return 0x923f82a4u; case 7: return 0xab1c5ed5u;
    case 8: return 0xd807aa98u; case 9: return 0x12835b01u; case 10: return 0x243185beu; case 11: return 0x550c7dc3u;
    case 12: return 0x72be5d74u; case 13: return 0x80deb1feu; case 14: return 0x9bdc06a7u; case 15: return 0xc19bf174u;
    case 16: return 0xe49b69c1u; case 17: return 0xefbe4786u; case 18: return 0x0fc19dc6u; case 19: return 0x240ca1ccu;
    case 20: return 0x2de92c6fu; case 21: return 0x4a7484aau; case 22: return 0x5cb0a9dcu; case 23: return 0x76f988dau;
    case 24: return 0x983e5152u; case 25: return 0xa831c66du; case 26: return 0xb00327c8u; case 27: return 0xbf597fc7u;
    case 28: return 0xc6e00bf3u; case 29: return 0xd5a79147u; case 30: return 0x06ca6351u; case 31: return 0x14292967u;
    case 32: return 0x27b70a85u; case 33: return 0x2e1b2138u; case 34: return 0x4d2c6dfcu; case 35: return 0x53380d13u;
    case 36: return 0x650a7354u; case 37: return 0x766a0abbu; case 38: return 0x81c2c92eu; case 39: return 0x92722c85u;
    case 40: return 0xa2bfe8a1u; case 41: return 0xa81a664bu; case 42: return 0xc24b8b70u; case 43: return 0xc76c51a3u;
    case 44: return 0xd192e819u; case 45: return 0xd6990624u; case 46: return 0xf40e3585u; case 47: return 0x106aa070u;
    case 48: return 0x19a4c116u; case 49: return 0x1e376c08u; case 50: return 0x2748774cu; case 51: return 0x34b0bcb5u;
    case 52: return 0x391c0cb3u; case 53: return 0x4ed8aa4au; case 54: return 0x5b9cca4fu; case 55: return 0x682e6ff3u;
    case 56: return 0x748f82eeu; case 57: return 0x78a5636fu; case 58: return 0x84c87814u; case 59: return 0x8cc70208u;
    case 60: return 0x90befffau; case 61: return 0xa4506cebu; case 62: return 0xbef9a3f7u; default: return 0xc67178f2u;
    }
}

// FIPS 180-4 section 5.3.3: initial hash value H(0).
__device__ __forceinline__ void sha_iv(uint32_t s[8]) {
    s[0] = 0x6a09e667u; s[1] = 0xbb67ae85u; s[2] = 0x3c6ef372u; s[3] = 0xa54ff53au;
    s[4] = 0x510e527fu; s[5] = 0x9b05688cu; s[6] = 0x1f83d9abu; s[7] = 0x5be0cd19u;
}

__device__ __forceinline__ uint32_t rotr(uint32_t x, int n) { return __funnelshift_r(x, x, n); }

// LOP3 truth tables over (a = 0xF0, b = 0xCC, c = 0xAA).
__device__ __forceinline__ uint32_t xor3(uint32_t a, uint32_t b, uint32_t c) {
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0x96;" : "=r"(r) : "r"(a), "r"(b), "r"(c));
    return r;
}
// Ch(x, y, z) = (x & y) ^ (~x & z)
__device__ __forceinline__ uint32_t ch(uint32_t x, uint32_t y, uint32_t z) {
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0xCA;" : "=r"(r) : "r"(x), "r"(y), "r"(z));
    return r;
}
// Maj(x, y, z) = (x & y) ^ (x & z) ^ (y & z)
__device__ __forceinline__ uint32_t maj(uint32_t x, uint32_t y, uint32_t z) {
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0xE8;" : "=r"(r) : "r"(x), "r"(y), "r"(z));
    return r;
}

__device__ __forceinline__ uint32_t bsig0(uint32_t x) { return xor3(rotr(x, 2), rotr(x, 13), rotr(x, 22)); }
__device__ __forceinline__ uint32_t bsig1(uint32_t x) { return xor3(rotr(x, 6), rotr(x, 11), rotr(x, 25)); }
__device__ __forceinline__ uint32_t ssig0(uint32_t x) { return xor3(rotr(x, 7), rotr(x, 18), x >> 3); }
__device__ __forceinline__ uint32_t ssig1(uint32_t x) { return xor3(rotr(x, 17), rotr(x, 19), x >> 10); }

// Big-endian word from 4 little-endian-loaded bytes, and back.
__device__ __forceinline__ uint32_t bswap32(uint32_t x) { return __byte_perm(x, 0u, 0x0123u); }

// Adders.  Every 32-bit add of the compression goes through one of these.
// AddAlu is a plain add (the compiler emits IADD3, mostly on the integer
// ALU pipe, the pipe that also carries every SHF and LOP3).  AddFma issues
// the add as IMAD a * one + b, with `one` a runtime 1 so that the compiler
// cannot turn the multiply-add back into an ALU add: IMAD goes to the FMA
// pipe.  Only the integer microbenchmark (int_peak.cu) uses it: SHA-256 with
// its adds moved there ran slower than with plain adds.
struct AddAlu {
    __device__ __forceinline__ uint32_t operator()(uint32_t a, uint32_t b) const { return a + b; }
};
struct AddFma {
    uint32_t one;
    __device__ __forceinline__ uint32_t operator()(uint32_t a, uint32_t b) const {
        uint32_t r;
        asm("mad.lo.u32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(one), "r"(b));
        return r;
    }
};

// One compression (FIPS 180-4 section 6.2.2, steps 1-4) of the 512-bit block
// w[0..15] (big-endian words) into the chaining state s.  w is overwritten by
// the message schedule.  CONST_W: w is a compile-time constant (a padding
// block), so its schedule and K_t + W_t are computed with plain operations
// and fold to immediates.  FROM_IV: s is the initial hash value, so round 0
// (all state words constant) also folds.
template <bool CONST_W, bool FROM_IV, class Add>
__device__ __forceinline__ void sha_compress_t(uint32_t s[8], uint32_t w[16], Add add) {
    uint32_t a = s[0], b = s[1], c = s[2], d = s[3];
    uint32_t e = s[4], f = s[5], g = s[6], h = s[7];
#pragma unroll
    for (int t = 0; t < 64; ++t) {
        const int i = t & 15;
        if (t >= 16) {
            if (CONST_W)
                w[i] += ssig1(w[(t - 2) & 15]) + w[(t - 7) & 15] + ssig0(w[(t - 15) & 15]);
            else
                w[i] = add(add(w[i], w[(t - 7) & 15]), add(ssig0(w[(t - 15) & 15]), ssig1(w[(t - 2) & 15])));
        }
        uint32_t t1, t2;
        if (FROM_IV && t == 0) {            // every state word is a constant
            t1 = h + sha_k(0) + ch(e, f, g) + bsig1(e) + w[0];
            t2 = bsig0(a) + maj(a, b, c);
            h = g; g = f; f = e; e = d + t1;
            d = c; c = b; b = a; a = t1 + t2;
            continue;
        }
        const uint32_t kw = CONST_W ? sha_k(t) + w[i] : add(w[i], sha_k(t));
        t1 = add(add(add(h, kw), ch(e, f, g)), bsig1(e));
        t2 = add(bsig0(a), maj(a, b, c));
        h = g; g = f; f = e; e = add(d, t1);
        d = c; c = b; b = a; a = add(t1, t2);
    }
    s[0] = add(s[0], a); s[1] = add(s[1], b); s[2] = add(s[2], c); s[3] = add(s[3], d);
    s[4] = add(s[4], e); s[5] = add(s[5], f); s[6] = add(s[6], g); s[7] = add(s[7], h);
}

template <class Add = AddAlu>
__device__ __forceinline__ void sha_compress(uint32_t s[8], uint32_t w[16], Add add = Add()) {
    sha_compress_t<false, false>(s, w, add);
}

// FIPS 180-4 section 4.2.2 K_t: in constant memory for the compact
// compression below, and as a host-side array for schedules the host
// computes ahead (a fixed padding block's).
#define KVGOV_SHA256_K \
    0x428a2f98u, 0x71374491u, 0xb5c0fbcfu, 0xe9b5dba5u, 0x3956c25bu, 0x59f111f1u, 0x923f82a4u, 0xab1c5ed5u, \
    0xd807aa98u, 0x12835b01u, 0x243185beu, 0x550c7dc3u, 0x72be5d74u, 0x80deb1feu, 0x9bdc06a7u, 0xc19bf174u, \
    0xe49b69c1u, 0xefbe4786u, 0x0fc19dc6u, 0x240ca1ccu, 0x2de92c6fu, 0x4a7484aau, 0x5cb0a9dcu, 0x76f988dau, \
    0x983e5152u, 0xa831c66du, 0xb00327c8u, 0xbf597fc7u, 0xc6e00bf3u, 0xd5a79147u, 0x06ca6351u, 0x14292967u, \
    0x27b70a85u, 0x2e1b2138u, 0x4d2c6dfcu, 0x53380d13u, 0x650a7354u, 0x766a0abbu, 0x81c2c92eu, 0x92722c85u, \
    0xa2bfe8a1u, 0xa81a664bu, 0xc24b8b70u, 0xc76c51a3u, 0xd192e819u, 0xd6990624u, 0xf40e3585u, 0x106aa070u, \
    0x19a4c116u, 0x1e376c08u, 0x2748774cu, 0x34b0bcb5u, 0x391c0cb3u, 0x4ed8aa4au, 0x5b9cca4fu, 0x682e6ff3u, \
    0x748f82eeu, 0x78a5636fu, 0x84c87814u, 0x8cc70208u, 0x90befffau, 0xa4506cebu, 0xbef9a3f7u, 0xc67178f2u
static __constant__ uint32_t c_sha_k[64] = {KVGOV_SHA256_K};
constexpr uint32_t kShaKHost[64] = {KVGOV_SHA256_K};

// The same compression with a small instruction footprint: rounds 0-15 are
// unrolled, rounds 16-63 run as three passes of one unrolled 16-round body
// (after 16 rounds the eight working variables are back in their original
// roles, so the loop carries them without moves), with K_t read from
// constant memory.  About a quarter of the code of sha_compress, for kernels
// whose time goes to instruction fetch rather than to the integer pipe.
template <class Add = AddAlu>
__device__ __forceinline__ void sha_compress_small(uint32_t s[8], uint32_t w[16], Add add = Add()) {
    uint32_t v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = s[i];
#pragma unroll
    for (int t = 0; t < 16; ++t) {
        uint32_t &a = v[(8 - t % 8) % 8], &b = v[(9 - t % 8) % 8], &c = v[(10 - t % 8) % 8], &d = v[(11 - t % 8) % 8];
        uint32_t &e = v[(12 - t % 8) % 8], &f = v[(13 - t % 8) % 8], &g = v[(14 - t % 8) % 8], &h = v[(15 - t % 8) % 8];
        const uint32_t t1 = add(add(add(h, add(w[t], sha_k(t))), ch(e, f, g)), bsig1(e));
        const uint32_t t2 = add(bsig0(a), maj(a, b, c));
        d = add(d, t1);
        h = add(t1, t2);
    }
#pragma unroll 1
    for (int base = 16; base < 64; base += 16) {
#pragma unroll
        for (int t = 0; t < 16; ++t) {
            w[t] = add(add(w[t], w[(t + 9) & 15]), add(ssig0(w[(t + 1) & 15]), ssig1(w[(t + 14) & 15])));
            uint32_t &a = v[(8 - t % 8) % 8], &b = v[(9 - t % 8) % 8], &c = v[(10 - t % 8) % 8], &d = v[(11 - t % 8) % 8];
            uint32_t &e = v[(12 - t % 8) % 8], &f = v[(13 - t % 8) % 8], &g = v[(14 - t % 8) % 8], &h = v[(15 - t % 8) % 8];
            const uint32_t t1 = add(add(add(h, add(w[t], c_sha_k[base + t])), ch(e, f, g)), bsig1(e));
            const uint32_t t2 = add(bsig0(a), maj(a, b, c));
            d = add(d, t1);
            h = add(t1, t2);
        }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i] = add(s[i], v[i]);
}

// sha_compress_small with the adds that are off the rounds' dependency chain
// issued on the FMA pipe (`side`, an IMAD with a run-time 1), which SHA-256
// otherwise leaves idle, so that the integer ALU pipe -- which alone runs the
// funnel shifts and three-input booleans -- carries fewer instructions:
//   hk = h + K_t + W_t and dk = d + hk, both known rounds ahead (h and d are
//   the e and a of three rounds before); then e' = dk + Ch + Sigma1 and
//   a' = (hk + Ch + Sigma1) + Sigma0 + Maj on the ALU;
//   in the schedule, W_t + W_{t-7} (known seven rounds ahead) on the FMA
//   pipe, then + sigma0 + sigma1 on the ALU; the final state adds too.
// The same sums in another grouping: the same digest.
__device__ __forceinline__ void sha_compress_small_split(uint32_t s[8], uint32_t w[16], AddFma side) {
    uint32_t v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = s[i];
#pragma unroll
    for (int t = 0; t < 16; ++t) {
        uint32_t &a = v[(8 - t % 8) % 8], &b = v[(9 - t % 8) % 8], &c = v[(10 - t % 8) % 8], &d = v[(11 - t % 8) % 8];
        uint32_t &e = v[(12 - t % 8) % 8], &f = v[(13 - t % 8) % 8], &g = v[(14 - t % 8) % 8], &h = v[(15 - t % 8) % 8];
        const uint32_t hk = side(h, side(w[t], sha_k(t)));
        const uint32_t dk = side(d, hk);
        const uint32_t cs = ch(e, f, g), s1 = bsig1(e);
        d = dk + cs + s1;
        h = (hk + cs + s1) + bsig0(a) + maj(a, b, c);
    }
#pragma unroll 1
    for (int base = 16; base < 64; base += 16) {
#pragma unroll
        for (int t = 0; t < 16; ++t) {
            w[t] = side(w[t], w[(t + 9) & 15]) + ssig0(w[(t + 1) & 15]) + ssig1(w[(t + 14) & 15]);
            uint32_t &a = v[(8 - t % 8) % 8], &b = v[(9 - t % 8) % 8], &c = v[(10 - t % 8) % 8], &d = v[(11 - t % 8) % 8];
            uint32_t &e = v[(12 - t % 8) % 8], &f = v[(13 - t % 8) % 8], &g = v[(14 - t % 8) % 8], &h = v[(15 - t % 8) % 8];
            const uint32_t hk = side(h, side(w[t], c_sha_k[base + t]));
            const uint32_t dk = side(d, hk);
            const uint32_t cs = ch(e, f, g), s1 = bsig1(e);
            d = dk + cs + s1;
            h = (hk + cs + s1) + bsig0(a) + maj(a, b, c);
        }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i] = side(s[i], v[i]);
}

// 16 rounds (FIPS 180-4 section 6.2.2 step 3) with K_t + W_t given, for
// kernels whose message schedule is computed elsewhere.  v holds a..h in
// rotating roles; after 16 rounds every variable is back in its original
// slot.  Two groupings of the same sums:
//   sha_rounds16_t1t2: T1 = h + KW + Ch + Sigma1, T2 = Sigma0 + Maj,
//                      e' = d + T1, a' = T1 + T2;
//   sha_rounds16_short: x = h + KW + Ch, e' = d + x + Sigma1 (one three-input
//                      add after Sigma1), a' = x + Sigma1 + Sigma0 + Maj;
// the second puts one add fewer between e and the next e.
__device__ __forceinline__ void sha_rounds16_t1t2(uint32_t v[8], const uint32_t kw[16]) {
#pragma unroll
    for (int t = 0; t < 16; ++t) {
        uint32_t &a = v[(8 - t % 8) % 8], &b = v[(9 - t % 8) % 8], &c = v[(10 - t % 8) % 8], &d = v[(11 - t % 8) % 8];
        uint32_t &e = v[(12 - t % 8) % 8], &f = v[(13 - t % 8) % 8], &g = v[(14 - t % 8) % 8], &h = v[(15 - t % 8) % 8];
        const uint32_t t1 = h + kw[t] + ch(e, f, g) + bsig1(e);
        const uint32_t t2 = bsig0(a) + maj(a, b, c);
        d += t1;
        h = t1 + t2;
    }
}
__device__ __forceinline__ void sha_rounds16_short(uint32_t v[8], const uint32_t kw[16]) {
#pragma unroll
    for (int t = 0; t < 16; ++t) {
        uint32_t &a = v[(8 - t % 8) % 8], &b = v[(9 - t % 8) % 8], &c = v[(10 - t % 8) % 8], &d = v[(11 - t % 8) % 8];
        uint32_t &e = v[(12 - t % 8) % 8], &f = v[(13 - t % 8) % 8], &g = v[(14 - t % 8) % 8], &h = v[(15 - t % 8) % 8];
        const uint32_t x = h + kw[t] + ch(e, f, g);
        const uint32_t s1 = bsig1(e);
        const uint32_t y = x + s1 + bsig0(a);
        d = d + x + s1;
        h = y + maj(a, b, c);
    }
}

// Compression of a data block inside the fixed-length messages below: the
// compact form (measured faster for the chain kernel on GB300, whose fully
// unrolled form stalls on instruction fetch).
template <bool FROM_IV, class Add>
__device__ __forceinline__ void sha_compress_data(uint32_t s[8], uint32_t w[16], Add add) {
    sha_compress_small(s, w, add);
}

// Fixed-length messages of the chain (section 2.1 / 4.1 / 4.2 equations).
// Arguments are big-endian message words; out gets the digest's state words
// (digest byte 4i.. 4i+3 = out[i] big-endian).  SHA-256 padding (section
// 5.1.1) appends 0x80, zeros and the 64-bit bit length; for these lengths the
// padding words are compile-time constants.

__device__ __forceinline__ void pad_block(uint32_t w[16], int first, uint32_t bits) {
#pragma unroll
    for (int i = 0; i < 16; ++i) w[i] = 0u;
    w[first] = 0x80000000u;
    w[15] = bits;
}

// H(T): 64-byte message = one data block + one constant padding block.
template <class Add>
__device__ __forceinline__ void sha256_msg64(const uint32_t tw[16], uint32_t out[8], Add add) {
    uint32_t s[8], w[16];
    sha_iv(s);
#pragma unroll
    for (int i = 0; i < 16; ++i) w[i] = tw[i];
    sha_compress_data<true>(s, w, add);
    pad_block(w, 0, 64u * 8u);
    sha_compress_t<true, false>(s, w, add);
#pragma unroll
    for (int i = 0; i < 8; ++i) out[i] = s[i];
}

// H(P || T): 32-byte prefix P (parent digest or salt) + 64-byte block.
template <class Add>
__device__ __forceinline__ void sha256_msg96(const uint32_t pw[8], const uint32_t tw[16], uint32_t out[8], Add add) {
    uint32_t s[8], w[16];
    sha_iv(s);
#pragma unroll
    for (int i = 0; i < 8; ++i) { w[i] = pw[i]; w[8 + i] = tw[i]; }
    sha_compress_data<true>(s, w, add);
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = tw[8 + i];
    w[8] = 0x80000000u;
#pragma unroll
    for (int i = 9; i < 15; ++i) w[i] = 0u;
    w[15] = 96u * 8u;
    sha_compress_data<false>(s, w, add);
#pragma unroll
    for (int i = 0; i < 8; ++i) out[i] = s[i];
}

// H(S || P || T): salt, parent digest, block (the boundary block of 4.2).
template <class Add>
__device__ __forceinline__ void sha256_msg128(const uint32_t sw[8], const uint32_t pw[8], const uint32_t tw[16],
                                              uint32_t out[8], Add add) {
    uint32_t s[8], w[16];
    sha_iv(s);
#pragma unroll
    for (int i = 0; i < 8; ++i) { w[i] = sw[i]; w[8 + i] = pw[i]; }
    sha_compress_data<true>(s, w, add);
#pragma unroll
    for (int i = 0; i < 16; ++i) w[i] = tw[i];
    sha_compress_data<false>(s, w, add);
    pad_block(w, 0, 128u * 8u);
    sha_compress_t<true, false>(s, w, add);
#pragma unroll
    for (int i = 0; i < 8; ++i) out[i] = s[i];
}

}  // namespace kvgov_dev
