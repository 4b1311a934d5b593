// Batch verification Pi_Batch-vMVMD (Protocol 2 of the paper): the client's
// checks, and the transposes the lane encoder needs.
//
//  * k_transpose_u32   out[c][r] = in[r][c] through 32 x 32 shared tiles.
//  * k_bv_checks       one CTA per check:
//                        (q, j) secondary: e^(q)^T Qaux e'^(j) == r^(j)^T u^(q)
//                               (t t' entries of Qaux, one length-B n dot)
//                        (b, q) original:  u_b^(q)^T x_b == e^(q)^T z_b
//                               (one length-n dot, t entries of z_b)
//                      a failed check clears the batch's accept flag.
#include "common.cuh"
#include "launch.h"

namespace pv {
namespace {

constexpr int kBvThreads = 256;

__global__ void k_transpose_u32(const uint32_t *__restrict__ in, int R, int C, uint32_t *__restrict__ out) {
    __shared__ uint32_t tile[32][33];
    const int c = blockIdx.x * 32 + threadIdx.x;
    for (int i = threadIdx.y; i < 32; i += 8) {
        const int r = blockIdx.y * 32 + i;
        if (r < R && c < C) tile[i][threadIdx.x] = in[(size_t)r * C + c];
    }
    __syncthreads();
    const int r = blockIdx.y * 32 + threadIdx.x;
    for (int i = threadIdx.y; i < 32; i += 8) {
        const int cc = blockIdx.x * 32 + i;
        if (r < R && cc < C) out[(size_t)cc * R + r] = tile[threadIdx.x][i];
    }
}

// Sum over the CTA of a value per thread, mod q; the result in every thread.
__device__ __forceinline__ uint32_t block_fsum(uint32_t v, uint32_t *red) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v = fadd(v, __shfl_xor_sync(kFull, v, o));
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    uint32_t s = 0;
    for (int w = 0; w < kBvThreads / 32; ++w) s = fadd(s, red[w]);
    return s;
}

__global__ void __launch_bounds__(kBvThreads) k_bv_checks(
    const uint32_t *__restrict__ QauxT, int N, int Bn, int n, int B, const uint32_t *__restrict__ chal,
    uint32_t t, uint32_t ell, const uint32_t *__restrict__ chal2, uint32_t t2, uint32_t ell2,
    const uint32_t *__restrict__ u, const uint32_t *__restrict__ R, const uint32_t *__restrict__ X,
    const uint32_t *__restrict__ Z, int32_t *accept) {
    __shared__ uint32_t red[kBvThreads / 32];
    const uint32_t blk = blockIdx.x, tid = threadIdx.x;
    uint64_t lhs = 0, rhs = 0;
    if (blk < ell * ell2) {  // secondary check (q, j)
        const uint32_t q = blk / ell2, j = blk % ell2;
        const uint32_t *s1 = chal + (size_t)q * 2 * t, *v1 = s1 + t;
        const uint32_t *s2 = chal2 + (size_t)j * 2 * t2, *v2 = s2 + t2;
        for (uint32_t idx = tid; idx < t * t2; idx += kBvThreads) {
            const uint32_t a = idx / t2, c = idx % t2;
            const uint32_t w = fmul(v1[a], v2[c]);
            lhs = fred(lhs + (uint64_t)w * QauxT[(size_t)s2[c] * N + s1[a]]);
        }
        const uint32_t *uq = u + (size_t)q * Bn, *rj = R + (size_t)j * Bn;
        for (int p = tid; p < Bn; p += kBvThreads) rhs = fred(rhs + (uint64_t)rj[p] * uq[p]);
    } else {  // original check (b, q)
        const uint32_t k = blk - ell * ell2, b = k / ell, q = k % ell;
        const uint32_t *ub = u + (size_t)q * Bn + (size_t)b * n, *xb = X + (size_t)b * n;
        for (int p = tid; p < n; p += kBvThreads) lhs = fred(lhs + (uint64_t)ub[p] * xb[p]);
        const uint32_t *s1 = chal + (size_t)q * 2 * t, *v1 = s1 + t;
        for (uint32_t a = tid; a < t; a += kBvThreads) rhs = fred(rhs + (uint64_t)v1[a] * Z[(size_t)s1[a] * B + b]);
    }
    const uint32_t L = block_fsum((uint32_t)lhs, red);
    const uint32_t Rv = block_fsum((uint32_t)rhs, red);
    if (tid == 0 && L != Rv) atomicAnd(accept, 0);
}

__global__ void k_set_i32(int32_t *p, int32_t v) { *p = v; }

}  // namespace

cudaError_t launch_transpose_u32(const uint32_t *in, int R, int C, uint32_t *out, cudaStream_t s) {
    if (R <= 0 || C <= 0) return cudaSuccess;
    dim3 grid((C + 31) / 32, (R + 31) / 32), block(32, 8);
    if (grid.y > 65535u) return cudaErrorInvalidValue;
    k_transpose_u32<<<grid, block, 0, s>>>(in, R, C, out); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_bv_checks(const uint32_t *QauxT, int N, int Bn, int n, int B, const uint32_t *chal,
                             uint32_t t, uint32_t ell, const uint32_t *chal2, uint32_t t2, uint32_t ell2,
                             const uint32_t *u, const uint32_t *R, const uint32_t *X, const uint32_t *Z,
                             int32_t *accept, cudaStream_t s) {
    k_set_i32<<<1, 1, 0, s>>>(accept, 1); note_launch();
    const size_t blocks = (size_t)ell * ell2 + (size_t)B * ell;
    if (blocks == 0) return cudaGetLastError();
    if (blocks > 0x7fffffffu) return cudaErrorInvalidValue;
    k_bv_checks<<<(unsigned)blocks, kBvThreads, 0, s>>>(QauxT, N, Bn, n, B, chal, t, ell, chal2, t2, ell2, u,
                                                        R, X, Z, accept); note_launch();
    return cudaGetLastError();
}

}  // namespace pv
