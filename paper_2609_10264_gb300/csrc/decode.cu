// Client decode and verification (Protocol 3, Verify and Decrypt).
//
//  * k_verify_u         u_q = e_q^T Q for the ell shared challenges
//                       (sum of t_y rows of Q, cost (2t-1)n per repetition,
//                       the e^T Q row of the cost table in Sec. 5.3).
//  * k_decode_verify    one thread-block cluster per vector b:
//                         Y_b = y_hat_b - P e_x,b   (t_x rows of P^T)
//                         L_q = u_q . x_hat_b,  R_q = g_q . y_hat_b
//                       where g_q = G_y e_q, so that
//                       R_q = e_q^T (G_y^T y_hat_b) by transposition;
//                       the CTAs of the cluster reduce their partial dot
//                       products through distributed shared memory and
//                       rank 0 writes accept_b = AND_q (L_q == R_q).
//                       In boost mode (Sec. 7.2) P e_x,b was prepared ahead
//                       and is read instead of the t_x rows of P^T.
//  * k_output_mask      the output masks P e_x,b alone (boost mode's
//                       offline step).
#include <cooperative_groups.h>

#include "common.cuh"
#include "launch.h"

namespace cg = cooperative_groups;

namespace pv {
namespace {

constexpr int kDecThreads = 256;
constexpr int kMaxEll = 16;

__device__ __forceinline__ uint4 ldg4(const uint32_t *p) {
    return __ldg(reinterpret_cast<const uint4 *>(p));
}

__global__ void __launch_bounds__(256) k_verify_u(const uint32_t *__restrict__ Qm, int K,
                                                 const uint32_t *__restrict__ chal, uint32_t t,
                                                 uint32_t *__restrict__ u) {
    extern __shared__ uint32_t sm[];
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");  // the challenges come from the kernel before
    const uint32_t q = blockIdx.y;
    const uint32_t *c = chal + (size_t)q * 2 * t;
    for (uint32_t j = threadIdx.x; j < 2 * t; j += blockDim.x) sm[j] = c[j];
    __syncthreads();
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    uint64_t acc = 0;
    uint32_t j = 0;
    for (; j + 8 <= t; j += 8) {
        uint32_t v[8];
#pragma unroll
        for (int s2 = 0; s2 < 8; ++s2) v[s2] = __ldg(Qm + (size_t)sm[j + s2] * K + k);
#pragma unroll
        for (int s2 = 0; s2 < 4; ++s2) acc += (uint64_t)sm[t + j + s2] * v[s2];
        acc = fred(acc);
#pragma unroll
        for (int s2 = 4; s2 < 8; ++s2) acc += (uint64_t)sm[t + j + s2] * v[s2];
        acc = fred(acc);
    }
    for (; j < t; ++j) acc = fred(acc + (uint64_t)sm[t + j] * __ldg(Qm + (size_t)sm[j] * K + k));
    u[(size_t)q * K + k] = (uint32_t)acc;
}

__device__ __forceinline__ uint32_t warp_fsum(uint32_t v) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v = fadd(v, __shfl_xor_sync(kFull, v, o));
    return v;
}

// pe[s] = sum_j vals[j] P^T[supp[j]][i + s] mod q for the four columns
// i .. i+3 (columns at or past c1 read as 0); 16-byte loads when vec.
__device__ __forceinline__ void pe_cols(const uint32_t *__restrict__ PT, int m, const uint32_t *supp,
                                    const uint32_t *vals, uint32_t t_x, int i, int c1, bool vec,
                                    uint32_t pe[4]) {
    uint64_t a0 = 0, a1 = 0, a2 = 0, a3 = 0;
    uint32_t j = 0;
    for (; j + 8 <= t_x; j += 8) {
        uint4 v[8];
#pragma unroll
        for (int s = 0; s < 8; ++s) {
            const uint32_t *row = PT + (size_t)supp[j + s] * m + i;
            if (vec) {
                v[s] = ldg4(row);
            } else {
                v[s].x = row[0];
                v[s].y = i + 1 < c1 ? row[1] : 0u;
                v[s].z = i + 2 < c1 ? row[2] : 0u;
                v[s].w = i + 3 < c1 ? row[3] : 0u;
            }
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
#pragma unroll
            for (int s = 4 * h; s < 4 * h + 4; ++s) {
                const uint64_t e = vals[j + s];
                a0 += e * v[s].x; a1 += e * v[s].y; a2 += e * v[s].z; a3 += e * v[s].w;
            }
            a0 = fred(a0); a1 = fred(a1); a2 = fred(a2); a3 = fred(a3);
        }
    }
    for (; j + 4 <= t_x; j += 4) {
        uint4 v[4];
#pragma unroll
        for (int s = 0; s < 4; ++s) {
            const uint32_t *row = PT + (size_t)supp[j + s] * m + i;
            if (vec) {
                v[s] = ldg4(row);
            } else {
                v[s].x = row[0];
                v[s].y = i + 1 < c1 ? row[1] : 0u;
                v[s].z = i + 2 < c1 ? row[2] : 0u;
                v[s].w = i + 3 < c1 ? row[3] : 0u;
            }
        }
#pragma unroll
        for (int s = 0; s < 4; ++s) {
            const uint64_t e = vals[j + s];
            a0 += e * v[s].x; a1 += e * v[s].y; a2 += e * v[s].z; a3 += e * v[s].w;
        }
        a0 = fred(a0); a1 = fred(a1); a2 = fred(a2); a3 = fred(a3);
    }
    for (; j < t_x; ++j) {
        const uint32_t *row = PT + (size_t)supp[j] * m + i;
        const uint64_t e = vals[j];
        a0 += e * row[0];
        if (i + 1 < c1) a1 += e * row[1];
        if (i + 2 < c1) a2 += e * row[2];
        if (i + 3 < c1) a3 += e * row[3];
    }
    pe[0] = fred(a0);
    pe[1] = fred(a1);
    pe[2] = fred(a2);
    pe[3] = fred(a3);
}

template <bool kBoost>
__global__ void __launch_bounds__(kDecThreads) k_decode_verify(
    const uint32_t *__restrict__ PT, int m, int K, const uint32_t *__restrict__ st, uint32_t t_x,
    const uint32_t *__restrict__ Xhat, const uint32_t *Yhat, const uint32_t *__restrict__ g,
    const uint32_t *__restrict__ u, uint32_t ell, uint32_t *Y, int32_t *__restrict__ accept,
    bool vec, const uint32_t *__restrict__ mask) {
    cg::cluster_group cluster = cg::this_cluster();
    extern __shared__ uint32_t sm[];  // support[t_x], values[t_x]
    __shared__ uint32_t s_part[2 * kMaxEll];
    __shared__ uint32_t s_warp[kDecThreads / 32][2 * kMaxEll];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t rank = cluster.block_rank();
    const uint32_t C = cluster.num_blocks();
    const size_t b = blockIdx.y;

    // Inputs of this kernel (P^T, st, x_hat, y_hat) were written before the
    // challenge kernels that precede it in the stream; g and u come from
    // those kernels, so they are read only after griddepcontrol.wait.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (!kBoost) {
        const uint32_t *stb = st + b * 2 * t_x;
        for (uint32_t j = tid; j < 2 * t_x; j += kDecThreads) sm[j] = stb[j];
    }
    uint32_t *ystage = sm + 2 * t_x;  // this CTA's y_hat columns (y may alias y_hat)
    __syncthreads();
    const uint32_t *supp = sm, *vals = sm + t_x;

    uint64_t racc[kMaxEll], lacc[kMaxEll];
#pragma unroll
    for (int q = 0; q < kMaxEll; ++q) racc[q] = lacc[q] = 0;

    // ---- decrypt and the y_hat side of the check over this CTA's columns
    const int chunk = (((m + (int)C - 1) / (int)C) + 3) & ~3;
    const int c0 = (int)rank * chunk;
    const int c1 = min(m, c0 + chunk);
    const uint32_t *yh = Yhat + b * m;
    uint32_t *yo = Y + b * m;
    for (int i = c0 + tid * 4; i < c1; i += kDecThreads * 4) {
        uint32_t pe[4];
        if (kBoost) {
#pragma unroll
            for (int q2 = 0; q2 < 4; ++q2) pe[q2] = i + q2 < c1 ? mask[b * m + i + q2] : 0u;
        } else {
            pe_cols(PT, m, supp, vals, t_x, i, c1, vec, pe);
        }

#pragma unroll
        for (int s = 0; s < 4; ++s) {
            const int col = i + s;
            if (col < c1) {
                const uint32_t yv = yh[col];
                ystage[col - c0] = yv;
                yo[col] = fsub(yv, pe[s]);
            }
        }
    }
    __syncthreads();
    asm volatile("griddepcontrol.wait;" ::: "memory");  // g and u are complete from here on
    int cnty = 0;
    for (int col = c0 + tid; col < c1; col += kDecThreads) {
        const uint64_t yv = ystage[col - c0];
        for (uint32_t q = 0; q < ell; ++q) racc[q] += (uint64_t)g[(size_t)q * m + col] * yv;
        if (++cnty == 4) {
            cnty = 0;
            for (uint32_t q = 0; q < ell; ++q) racc[q] = fred(racc[q]);
        }
    }

    // ---- the x_hat side over this CTA's slice of K
    const int kc = (K + (int)C - 1) / (int)C;
    const int k0 = (int)rank * kc, k1 = min(K, k0 + kc);
    const uint32_t *xh = Xhat + b * K;
    int cnt = 0;
    for (int k = k0 + tid; k < k1; k += kDecThreads) {
        const uint64_t xv = xh[k];
        for (uint32_t q = 0; q < ell; ++q) lacc[q] += (uint64_t)u[(size_t)q * K + k] * xv;
        if (++cnt == 4) {
            cnt = 0;
            for (uint32_t q = 0; q < ell; ++q) lacc[q] = fred(lacc[q]);
        }
    }

    for (uint32_t q = 0; q < ell; ++q) {
        const uint32_t l = warp_fsum(fred(lacc[q]));
        const uint32_t r = warp_fsum(fred(racc[q]));
        if (lane == 0) {
            s_warp[warp][q] = l;
            s_warp[warp][kMaxEll + q] = r;
        }
    }
    __syncthreads();
    if (tid < 2 * kMaxEll) {
        uint32_t s = 0;
        for (int w = 0; w < kDecThreads / 32; ++w) s = fadd(s, s_warp[w][tid]);
        s_part[tid] = s;
    }
    cluster.sync();
    if (rank == 0 && tid == 0) {
        int ok = 1;
        for (uint32_t q = 0; q < ell; ++q) {
            uint32_t L = 0, R = 0;
            for (uint32_t r = 0; r < C; ++r) {
                const uint32_t *rp = cluster.map_shared_rank(s_part, r);
                L = fadd(L, rp[q]);
                R = fadd(R, rp[kMaxEll + q]);
            }
            ok &= (L == R);
        }
        accept[b] = ok;
    }
    cluster.sync();
}

// out[b][col] = (P e_x,b)_col for the columns of this CTA (1024 per CTA).
__global__ void __launch_bounds__(kDecThreads) k_output_mask(const uint32_t *__restrict__ PT, int m,
                                                            const uint32_t *__restrict__ st, uint32_t t_x,
                                                            uint32_t *__restrict__ out, bool vec) {
    extern __shared__ uint32_t sm[];  // support[t_x], values[t_x]
    const size_t b = blockIdx.y;
    const uint32_t *stb = st + b * 2 * t_x;
    for (uint32_t j = threadIdx.x; j < 2 * t_x; j += kDecThreads) sm[j] = stb[j];
    __syncthreads();
    const int i = (int)blockIdx.x * kDecThreads * 4 + (int)threadIdx.x * 4;
    if (i >= m) return;
    uint32_t pe[4];
    pe_cols(PT, m, sm, sm + t_x, t_x, i, m, vec, pe);
#pragma unroll
    for (int s = 0; s < 4; ++s)
        if (i + s < m) out[b * m + i + s] = pe[s];
}

// out = a + b over F_q, n elements, 16 bytes per thread where aligned.
__global__ void __launch_bounds__(256) k_field_add(const uint32_t *a, const uint32_t *b, size_t n,
                                                  uint32_t *out, bool vec) {
    const size_t i = ((size_t)blockIdx.x * 256 + threadIdx.x) * 4;
    if (i >= n) return;
    if (vec && i + 4 <= n) {
        const uint4 x = *reinterpret_cast<const uint4 *>(a + i);
        const uint4 y = *reinterpret_cast<const uint4 *>(b + i);
        *reinterpret_cast<uint4 *>(out + i) = make_uint4(fadd(x.x, y.x), fadd(x.y, y.y), fadd(x.z, y.z), fadd(x.w, y.w));
    } else {
        for (size_t k = i; k < n && k < i + 4; ++k) out[k] = fadd(a[k], b[k]);
    }
}

}  // namespace

cudaError_t launch_field_add(const uint32_t *a, const uint32_t *b, size_t n, uint32_t *out,
                             cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const bool vec = ((reinterpret_cast<uintptr_t>(a) | reinterpret_cast<uintptr_t>(b) |
                       reinterpret_cast<uintptr_t>(out)) & 15u) == 0;
    const size_t blocks = (n + 1023) / 1024;
    if (blocks > 0x7fffffffu) return cudaErrorInvalidValue;
    k_field_add<<<(unsigned)blocks, 256, 0, s>>>(a, b, n, out, vec);
    return cudaGetLastError();
}

cudaError_t launch_output_mask(const uint32_t *PT, int m, const uint32_t *st, uint32_t t_x, int B,
                               uint32_t *out, cudaStream_t s) {
    if (B <= 0 || m <= 0) return cudaSuccess;
    const bool vec = (m % 4 == 0) && ((reinterpret_cast<uintptr_t>(PT) & 15u) == 0);
    for (int b0 = 0; b0 < B; b0 += 65535) {
        const int nb = B - b0 < 65535 ? B - b0 : 65535;
        dim3 grid((m + kDecThreads * 4 - 1) / (kDecThreads * 4), nb);
        k_output_mask<<<grid, kDecThreads, 2 * (size_t)t_x * sizeof(uint32_t), s>>>(
            PT, m, st + (size_t)b0 * 2 * t_x, t_x, out + (size_t)b0 * m, vec);
    }
    return cudaGetLastError();
}

cudaError_t launch_verify_u(const uint32_t *Qm, int K, const uint32_t *chal, uint32_t t_y,
                            uint32_t ell, uint32_t *u, cudaStream_t s) {
    if (K <= 0 || ell == 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((K + 255) / 256, ell, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.dynamicSmemBytes = 2 * (size_t)t_y * sizeof(uint32_t);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_verify_u, Qm, K, chal, t_y, u);
}

cudaError_t launch_decode_verify(const uint32_t *PT, int m, int K, const uint32_t *st, uint32_t t_x,
                                 const uint32_t *Xhat, const uint32_t *Yhat, const uint32_t *g,
                                 const uint32_t *u, uint32_t ell, int B, uint32_t *Y,
                                 int32_t *accept, cudaStream_t s, const uint32_t *mask) {
    if (B <= 0) return cudaSuccess;
    if (ell > (uint32_t)kMaxEll) return cudaErrorInvalidValue;
    const bool vec = (m % 4 == 0) && ((reinterpret_cast<uintptr_t>(PT) & 15u) == 0);
    int C = (m + 1023) / 1024;
    C = C < 1 ? 1 : (C > 8 ? 8 : C);
    const int chunk = (((m + C - 1) / C) + 3) & ~3;  // y_hat columns per CTA (staged in smem)
    if ((2 * (size_t)t_x + (size_t)chunk) * sizeof(uint32_t) > 200 * 1024) return cudaErrorInvalidValue;
    static const cudaError_t smem_attr = cudaFuncSetAttribute(
        k_decode_verify<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    static const cudaError_t smem_attr2 = cudaFuncSetAttribute(
        k_decode_verify<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    if (smem_attr != cudaSuccess) return smem_attr;
    if (smem_attr2 != cudaSuccess) return smem_attr2;
    for (int b0 = 0; b0 < B; b0 += 65535) {
        const int nb = B - b0 < 65535 ? B - b0 : 65535;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(C, nb, 1);
        cfg.blockDim = dim3(kDecThreads, 1, 1);
        cfg.dynamicSmemBytes = (2 * (size_t)t_x + (size_t)chunk) * sizeof(uint32_t);
        cfg.stream = s;
        cudaLaunchAttribute attr[2];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = C;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[1].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 2;
        cudaError_t e = mask ? cudaLaunchKernelEx(&cfg, k_decode_verify<true>, PT, m, K, st, t_x,
                                                  Xhat + (size_t)b0 * K, Yhat + (size_t)b0 * m, g, u,
                                                  ell, Y + (size_t)b0 * m, accept + b0, vec,
                                                  mask + (size_t)b0 * m)
                             : cudaLaunchKernelEx(&cfg, k_decode_verify<false>, PT, m, K,
                                                  st + (size_t)b0 * 2 * t_x, t_x, Xhat + (size_t)b0 * K,
                                                  Yhat + (size_t)b0 * m, g, u, ell, Y + (size_t)b0 * m,
                                                  accept + b0, vec, (const uint32_t *)nullptr);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

}  // namespace pv
