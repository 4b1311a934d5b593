// Device-side helpers shared by the pvMVMD kernels: BabyBear field arithmetic,
// the ChaCha20 block function, bounded waits and the device error word.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

#include "pvmvmd.h"

namespace pv {

constexpr uint32_t kQ = PVMVMD_Q;            // 15 * 2^27 + 1 (Sec. 7.1)
constexpr uint32_t kHalfQ = (PVMVMD_Q - 1) / 2;
constexpr unsigned kFull = 0xffffffffu;

// Bits OR-ed into the library's device error word.
enum : uint32_t {
    kErrScanTimeout = 1u,   // a decoupled look-back wait expired
    kErrMmaTimeout = 2u,    // a tensor-core pipeline barrier wait expired
};

// Bounded waits: iteration cap and back-off (a wait that expires records an
// error bit and lets the kernel finish instead of spinning forever).
constexpr uint32_t kSpinLimit = 1u << 22;

// ---------------------------------------------------------------- field F_q
__host__ __device__ __forceinline__ uint32_t fadd(uint32_t a, uint32_t b) {
    uint32_t r = a + b;  // a, b < q < 2^31, so no wrap
    return r >= kQ ? r - kQ : r;
}
__host__ __device__ __forceinline__ uint32_t fsub(uint32_t a, uint32_t b) {
    return a >= b ? a - b : a + (kQ - b);
}
// x mod q for any 64-bit x.  On the device by Barrett reduction (Barrett,
// CRYPTO 1986): with mu = floor(2^64 / q), est = floor(x mu / 2^64) is
// floor(x / q) or one less (the error x (2^64/q - mu) / 2^64 is below 1), so
// x - est q lies in [0, 2q) and one conditional subtraction finishes.
constexpr uint64_t kBarrettMu = 0xFFFFFFFFFFFFFFFFull / PVMVMD_Q;  // = floor(2^64 / q), q odd
__host__ __device__ __forceinline__ uint32_t fred(uint64_t v) {
#ifdef __CUDA_ARCH__
    const uint64_t est = __umul64hi(v, kBarrettMu);
    const uint64_t r = v - est * kQ;
    return (uint32_t)(r >= kQ ? r - kQ : r);
#else
    return (uint32_t)(v % kQ);
#endif
}
__host__ __device__ __forceinline__ uint32_t fmul(uint32_t a, uint32_t b) {
    return fred((uint64_t)a * b);
}
// Montgomery multiplication with R = 2^32 (Montgomery, Math. Comp. 1985):
// for a < q and b < q, mont(a, b) = a b R^-1 mod q.  With b_m = b R mod q
// stored in a table, mont(a, b_m) = a b, the canonical product, in a few
// integer instructions: t = a b_m; m = -t q^-1 mod 2^32; (t + m q) / 2^32 < 2q.
constexpr uint32_t qinv_mod_2_32() {
    uint32_t x = PVMVMD_Q;  // Newton: each step doubles the correct low bits
    for (int i = 0; i < 5; ++i) x *= 2u - PVMVMD_Q * x;
    return x;
}
constexpr uint32_t kQInvNeg = 0u - qinv_mod_2_32();
static_assert(PVMVMD_Q * qinv_mod_2_32() == 1u, "q^-1 mod 2^32");
__host__ __device__ __forceinline__ uint32_t fmul_mont(uint32_t a, uint32_t b_m) {
    const uint64_t t = (uint64_t)a * b_m;
    const uint32_t m = (uint32_t)t * kQInvNeg;
    const uint64_t u = (t + (uint64_t)m * kQ) >> 32;  // t + m q < 2^62 + 2^63
    return (uint32_t)(u >= kQ ? u - kQ : u);
}
// b -> b R mod q (host table preparation).
__host__ __device__ __forceinline__ uint32_t to_mont(uint32_t b) {
    return (uint32_t)(((uint64_t)b << 32) % kQ);
}

// Signed 64-bit integer -> canonical representative.
__host__ __device__ __forceinline__ uint32_t fred_signed(int64_t v) {
#ifdef __CUDA_ARCH__
    if (v >= 0) return fred((uint64_t)v);
    const uint32_t r = fred(0ull - (uint64_t)v);  // |v|, exact also for INT64_MIN
    return r ? kQ - r : 0u;
#else
    int64_t r = v % (int64_t)kQ;
    return (uint32_t)(r < 0 ? r + (int64_t)kQ : r);
#endif
}
__host__ __device__ __forceinline__ uint32_t flift_i8(int8_t w) {
    return w < 0 ? kQ + (uint32_t)(int32_t)w : (uint32_t)w;
}

// Canonical x in [0, q) -> centred c in [-(q-1)/2, (q-1)/2] -> four signed
// base-256 digits d0..d3 in [-128, 127] with c = d0 + 2^8 d1 + 2^16 d2 + 2^24 d3
// (|d3| <= 61 because |c| < 2^30).
__device__ __forceinline__ void limb_split(uint32_t x, int &d0, int &d1, int &d2, int &d3) {
    int c = x > kHalfQ ? (int)(x - kQ) : (int)x;
    d0 = (int)(int8_t)(c & 0xff);
    c = (c - d0) >> 8;
    d1 = (int)(int8_t)(c & 0xff);
    c = (c - d1) >> 8;
    d2 = (int)(int8_t)(c & 0xff);
    d3 = (c - d2) >> 8;
}

// ---------------------------------------------------------------- ChaCha20
// RFC 8439 Sec. 2.3 block function; state words 4..11 key, 12 counter,
// 13..15 nonce.
__device__ __forceinline__ void chacha_qr(uint32_t &a, uint32_t &b, uint32_t &c, uint32_t &d) {
    a += b; d ^= a; d = __funnelshift_l(d, d, 16);
    c += d; b ^= c; b = __funnelshift_l(b, b, 12);
    a += b; d ^= a; d = __funnelshift_l(d, d, 8);
    c += d; b ^= c; b = __funnelshift_l(b, b, 7);
}

__device__ __forceinline__ void chacha20_block_dev(const pvmvmd_key &key, uint32_t counter,
                                                   uint32_t n0, uint32_t n1, uint32_t n2,
                                                   uint32_t out[16]) {
    const uint32_t init[16] = {0x61707865u, 0x3320646eu, 0x79622d32u, 0x6b206574u,
                               key.k[0], key.k[1], key.k[2], key.k[3],
                               key.k[4], key.k[5], key.k[6], key.k[7],
                               counter, n0, n1, n2};
    uint32_t x[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) x[i] = init[i];
#pragma unroll 1
    for (int dr = 0; dr < 10; ++dr) {
        chacha_qr(x[0], x[4], x[8], x[12]);
        chacha_qr(x[1], x[5], x[9], x[13]);
        chacha_qr(x[2], x[6], x[10], x[14]);
        chacha_qr(x[3], x[7], x[11], x[15]);
        chacha_qr(x[0], x[5], x[10], x[15]);
        chacha_qr(x[1], x[6], x[11], x[12]);
        chacha_qr(x[2], x[7], x[8], x[13]);
        chacha_qr(x[3], x[4], x[9], x[14]);
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) out[i] = x[i] + init[i];
}

// ---------------------------------------------------------------- memory ordering
__device__ __forceinline__ void st_release_u64(unsigned long long *p, unsigned long long v) {
    asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
// Relaxed 64-bit accesses: an aligned 64-bit word is read and written whole,
// so a state and a value packed into one word need no fence between them.
__device__ __forceinline__ void st_relaxed_u64(unsigned long long *p, unsigned long long v) {
    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release_u32(uint32_t *p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t *p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t ld_cg_u32(const uint32_t *p) { return __ldcg(p); }

__device__ __forceinline__ void record_error(uint32_t *err, uint32_t bit) {
    if (err) atomicOr(err, bit);
}

__device__ __forceinline__ uint32_t lanemask_lt() {
    uint32_t m;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

}  // namespace pv
