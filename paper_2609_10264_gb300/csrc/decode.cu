// Client decode and verification (Protocol 3, Verify and Decrypt).
//
//  * k_verify_u         u_q = e_q^T Q for the ell shared challenges
//                       (sum of t_y rows of Q, cost (2t-1)n per repetition,
//                       the e^T Q row of the cost table in Sec. 5.3).
//  * k_decrypt          Y_b = y_hat_b - P e_x,b (t_x rows of P^T), many
//                       short CTAs: 512 columns of one vector each, the
//                       rows split over two groups; in boost mode
//                       (Sec. 7.2) P e_x,b was prepared ahead and is read
//                       instead of the t_x rows of P^T.
//  * k_check            accept_b = AND_q (L_q == R_q), L_q = u_q . x_hat_b,
//                       R_q = g_q . y_hat_b with g_q = G_y e_q, so that
//                       R_q = e_q^T (G_y^T y_hat_b) by transposition.
//  * k_output_mask      the output masks P e_x,b alone (boost mode's
//                       offline step).
#include <cmath>
#include <map>
#include <mutex>

#include "common.cuh"
#include "launch.h"

namespace pv {
namespace {

constexpr int kDecThreads = 256;

__device__ __forceinline__ uint4 ldg4(const uint32_t *p) {
    return __ldg(reinterpret_cast<const uint4 *>(p));
}

// u[q][k] = sum_j chal_val[q][j] Q[chal_supp[q][j]][k]: a CTA covers 64
// columns with the t rows split over four row groups (so a thread streams
// about t/4 rows, one round of loads for t = 31), the groups' sums meeting
// in shared memory.
constexpr int kVuCols = 64, kVuGroups = 4;
__global__ void __launch_bounds__(kVuCols * kVuGroups) k_verify_u(const uint32_t *__restrict__ Qm, int K,
                                                                 const uint32_t *__restrict__ chal, uint32_t t,
                                                                 uint32_t *__restrict__ u) {
    extern __shared__ uint32_t sm[];
    __shared__ uint32_t s_part[kVuGroups - 1][kVuCols];
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");  // the challenges come from the kernel before
    const uint32_t q = blockIdx.y;
    const int tid = threadIdx.x, grp = tid / kVuCols, c = tid % kVuCols;
    const uint32_t *ch = chal + (size_t)q * 2 * t;
    for (uint32_t j = tid; j < 2 * t; j += kVuCols * kVuGroups) sm[j] = ch[j];
    __syncthreads();
    const int k = blockIdx.x * kVuCols + c;
    const uint32_t per = (t + kVuGroups - 1) / kVuGroups;
    const uint32_t j0 = min(t, (uint32_t)grp * per), j1 = min(t, j0 + per);
    uint64_t acc = 0;
    if (k < K) {
        uint32_t j = j0;
        for (; j + 8 <= j1; j += 8) {
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
        for (; j < j1; ++j) acc = fred(acc + (uint64_t)sm[t + j] * __ldg(Qm + (size_t)sm[j] * K + k));
    }
    if (grp > 0) s_part[grp - 1][c] = (uint32_t)acc;
    __syncthreads();
    if (grp == 0 && k < K) {
        uint32_t sum = (uint32_t)acc;
#pragma unroll
        for (int g2 = 0; g2 < kVuGroups - 1; ++g2) sum = fadd(sum, s_part[g2][c]);
        u[(size_t)q * K + k] = sum;
    }
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

// ---------------------------------------------------------------------------
// Decrypt: Y_b = y_hat_b - P e_x,b.  A CTA owns 512 columns of one vector
// (128 column threads x 4 columns, so each row of P^T is read in 2 KiB
// segments) and splits the t_x rows over kDecGroups = 2 row groups, so each
// thread streams about t_x / 2 row segments (rounds of 8 loads in flight)
// and the grid holds many short CTAs whatever m and B are; or 256 columns
// over 4 row groups when that fills the last wave of resident CTAs better.
// The groups' partial sums meet in shared memory.  (256 columns everywhere,
// or 1024 columns and 1 group, were 6 and 13 % slower at m = K = 8192,
// B = 256.)
// In boost mode (Sec. 7.2) P e_x,b was prepared ahead: Y_b = y_hat_b - mask_b.
// The grid runs vectors fastest (blockIdx.x = b, blockIdx.y = column block),
// so the CTAs in flight share a few column blocks and a row of P^T drawn by
// several vectors' supports is read from HBM once and then from L2.
// ---------------------------------------------------------------------------
template <bool kBoost, int kDecGroups>
__global__ void __launch_bounds__(kDecThreads) k_decrypt(const uint32_t *__restrict__ PT, int m,
                                                        const uint32_t *__restrict__ st, uint32_t t_x,
                                                        uint32_t Nx, const uint32_t *Yhat, uint32_t *Y,
                                                        const uint32_t *__restrict__ mask, bool vec) {
    constexpr int kDecColThreads = kDecThreads / kDecGroups;
    constexpr int kDecCols = 4 * kDecColThreads;
    extern __shared__ uint32_t sm[];  // support[t_x], values[t_x]
    __shared__ uint4 s_part[kDecGroups > 1 ? kDecGroups - 1 : 1][kDecColThreads];
    const int tid = threadIdx.x;
    const size_t b = blockIdx.x;
    const int grp = tid / kDecColThreads, ct = tid % kDecColThreads;
    // boost mode: no rows to split, every thread owns 4 of 1024 columns
    const int i = kBoost ? ((int)blockIdx.y * kDecThreads + tid) * 4 : (int)blockIdx.y * kDecCols + ct * 4;
    uint32_t pe[4] = {0u, 0u, 0u, 0u};
    if (!kBoost) {
        const uint32_t *stb = st + b * 2 * t_x;
        // a support index past the code (a state the encode did not write)
        // reads row 0 instead: the result is then wrong, never out of bounds
        for (uint32_t j = tid; j < 2 * t_x; j += kDecThreads) {
            const uint32_t v = stb[j];
            sm[j] = (j < t_x && v >= Nx) ? 0u : v;
        }
        __syncthreads();
        const uint32_t per = (t_x + kDecGroups - 1) / kDecGroups;
        const uint32_t j0 = min(t_x, (uint32_t)grp * per), j1 = min(t_x, j0 + per);
        if (i < m && j0 < j1) pe_cols(PT, m, sm + j0, sm + t_x + j0, j1 - j0, i, m, vec, pe);
        if (grp > 0) s_part[grp - 1][ct] = make_uint4(pe[0], pe[1], pe[2], pe[3]);
        __syncthreads();
        if (grp > 0) return;
#pragma unroll
        for (int g2 = 0; g2 < kDecGroups - 1; ++g2) {
            const uint4 v = s_part[g2][ct];
            pe[0] = fadd(pe[0], v.x);
            pe[1] = fadd(pe[1], v.y);
            pe[2] = fadd(pe[2], v.z);
            pe[3] = fadd(pe[3], v.w);
        }
    }
    if (i >= m) return;
    const uint32_t *yh = Yhat + b * m;
    uint32_t *yo = Y + b * m;
    if (kBoost) {
        const uint32_t *mk = mask + b * m;
#pragma unroll
        for (int q2 = 0; q2 < 4; ++q2) pe[q2] = i + q2 < m ? mk[i + q2] : 0u;
    }
    if (vec) {
        // y_hat is read here rather than prefetched before the row loop: a
        // live uint4 across the loop raises the kernel to 70 registers and
        // four CTAs per SM to three
        const uint4 yv = *reinterpret_cast<const uint4 *>(yh + i);
        *reinterpret_cast<uint4 *>(yo + i) =
            make_uint4(fsub(yv.x, pe[0]), fsub(yv.y, pe[1]), fsub(yv.z, pe[2]), fsub(yv.w, pe[3]));
    } else {
#pragma unroll
        for (int q2 = 0; q2 < 4; ++q2)
            if (i + q2 < m) yo[i + q2] = fsub(yh[i + q2], pe[q2]);
    }
}

// ---------------------------------------------------------------------------
// Verify: accept_b = AND_q [ L_q == R_q ] with L_q = u_q . x_hat_b and
// R_q = g_q . y_hat_b (= e_q^T (G_y^T y_hat_b) by transposition), u_q =
// e_q^T Q and g_q = G_y e_q from the challenge kernels.  One CTA per vector;
// the repetitions run one after the other over the (cached) vectors.
// ---------------------------------------------------------------------------
// 512 threads with eight loads of each operand in flight (1024 threads with
// four, an SM's whole register file per CTA, waited longer for SMs beside
// the decrypts: 8B layer 0.500 -> 0.492 ms, 70B layer 2.218 -> 2.191 ms per
// step, the batch-1 workload unchanged at 0.320 ms; 256 threads were
// slower)
constexpr int kCheckThreads = 512;
constexpr int kCheckBatch = 8;  // loads in flight per operand and thread

__global__ void __launch_bounds__(kCheckThreads) k_check(const uint32_t *__restrict__ Xhat, int K,
                                                        const uint32_t *__restrict__ Yhat, int m,
                                                        const uint32_t *__restrict__ g,
                                                        const uint32_t *__restrict__ u, uint32_t ell,
                                                        int32_t *__restrict__ accept) {
    __shared__ uint32_t s_part[4][kCheckThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const size_t b = blockIdx.x;
    const uint32_t *xh = Xhat + b * K, *yh = Yhat + b * m;
    // the kernel after this one (the next call's encode) may start its
    // key-only work now
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int n = K > m ? K : m;
    int ok = 1;
    // two repetitions per pass: x_hat and y_hat are read once per pair
    for (uint32_t q = 0; q < ell; q += 2) {
        const bool two = q + 1 < ell;
        const uint32_t *u0 = u + (size_t)q * K, *g0 = g + (size_t)q * m;
        const uint32_t *u1 = two ? u0 + K : u0, *g1 = two ? g0 + m : g0;
        uint64_t l0 = 0, l1 = 0, r0 = 0, r1 = 0;
        for (int k0 = tid; k0 < n; k0 += kCheckBatch * kCheckThreads) {
            uint32_t x[kCheckBatch], y[kCheckBatch], a0[kCheckBatch], a1[kCheckBatch], c0[kCheckBatch],
                c1[kCheckBatch];
#pragma unroll
            for (int v = 0; v < kCheckBatch; ++v) {
                const int k = k0 + v * kCheckThreads;
                const bool kx = k < K, ky = k < m;
                x[v] = kx ? xh[k] : 0u;
                a0[v] = kx ? __ldg(u0 + k) : 0u;
                a1[v] = kx ? __ldg(u1 + k) : 0u;
                y[v] = ky ? yh[k] : 0u;
                c0[v] = ky ? __ldg(g0 + k) : 0u;
                c1[v] = ky ? __ldg(g1 + k) : 0u;
            }
            // four products of values below q stay below 2^64 with the
            // reduced running sum, so the sums are reduced every four
#pragma unroll
            for (int v0 = 0; v0 < kCheckBatch; v0 += 4) {
#pragma unroll
                for (int v = v0; v < v0 + 4; ++v) {
                    l0 += (uint64_t)a0[v] * x[v];
                    l1 += (uint64_t)a1[v] * x[v];
                    r0 += (uint64_t)c0[v] * y[v];
                    r1 += (uint64_t)c1[v] * y[v];
                }
                l0 = fred(l0);
                l1 = fred(l1);
                r0 = fred(r0);
                r1 = fred(r1);
            }
            static_assert(kCheckBatch % 4 == 0, "sums reduced every four products");
        }
        const uint32_t w0 = warp_fsum((uint32_t)l0), w1 = warp_fsum((uint32_t)l1);
        const uint32_t w2 = warp_fsum((uint32_t)r0), w3 = warp_fsum((uint32_t)r1);
        if (lane == 0) {
            s_part[0][warp] = w0;
            s_part[1][warp] = w1;
            s_part[2][warp] = w2;
            s_part[3][warp] = w3;
        }
        __syncthreads();
        if (tid == 0) {
            uint32_t L0 = 0, L1 = 0, R0 = 0, R1 = 0;
            for (int w = 0; w < kCheckThreads / 32; ++w) {
                L0 = fadd(L0, s_part[0][w]);
                L1 = fadd(L1, s_part[1][w]);
                R0 = fadd(R0, s_part[2][w]);
                R1 = fadd(R1, s_part[3][w]);
            }
            ok &= (L0 == R0);
            if (two) ok &= (L1 == R1);
        }
        __syncthreads();
    }
    if (tid == 0) accept[b] = ok;
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
    k_field_add<<<(unsigned)blocks, 256, 0, s>>>(a, b, n, out, vec); note_launch();
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
            PT, m, st + (size_t)b0 * 2 * t_x, t_x, out + (size_t)b0 * m, vec); note_launch();
    }
    return cudaGetLastError();
}

cudaError_t launch_verify_u(const uint32_t *Qm, int K, const uint32_t *chal, uint32_t t_y,
                            uint32_t ell, uint32_t *u, cudaStream_t s) {
    if (K <= 0 || ell == 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((K + kVuCols - 1) / kVuCols, ell, 1);
    cfg.blockDim = dim3(kVuCols * kVuGroups, 1, 1);
    cfg.dynamicSmemBytes = 2 * (size_t)t_y * sizeof(uint32_t);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return counted_launch(cudaLaunchKernelEx(&cfg, k_verify_u, Qm, K, chal, t_y, u));
}

// Resident k_decrypt CTAs on the current device (cached per device).
int decrypt_slots() {
    static std::mutex mu;
    static std::map<int, int> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
    }
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(dev);
    if (it != cache.end()) return it->second;
    int per_sm = 0, sms = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_decrypt<false, 2>, kDecThreads, 1024) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        (void)cudaGetLastError();
        per_sm = 0;
    }
    return cache[dev] = per_sm * sms;
}

cudaError_t launch_decrypt(const uint32_t *PT, int m, const uint32_t *st, uint32_t t_x, uint32_t Nx,
                           const uint32_t *Yhat, int B, uint32_t *Y, cudaStream_t s, const uint32_t *mask) {
    if (B <= 0 || m <= 0) return cudaSuccess;
    const bool vec = (m % 4 == 0) &&
                     ((reinterpret_cast<uintptr_t>(PT) | reinterpret_cast<uintptr_t>(Yhat) |
                       reinterpret_cast<uintptr_t>(Y)) & 15u) == 0;
    const size_t smem = mask ? 0 : 2 * (size_t)t_x * sizeof(uint32_t);
    if (smem > 48 * 1024) return cudaErrorInvalidValue;
    const dim3 grid_mask((unsigned)B, (m + 4 * kDecThreads - 1) / (4 * kDecThreads));
    if (mask) {
        k_decrypt<true, 2><<<grid_mask, kDecThreads, 0, s>>>(PT, m, nullptr, t_x, Nx, Yhat, Y, mask, vec);
        note_launch();
        return cudaGetLastError();
    }
    // Every CTA streams the same t_x row segments, so a last wave that is a
    // third full costs as much as a full one: 256-column CTAs are used when
    // they fill the last wave of resident CTAs clearly better than 512
    // (4096 x 4096, 100 vectors: 800 CTAs are 1.32 waves of 608, 1600 are
    // 2.63; decrypt 47 -> 41 us, step 0.3221 -> 0.3202 ms).  Where both
    // fill alike the wider CTAs stay (70B-class shapes, 256 vectors: 256
    // columns everywhere took 2.221 -> 2.272 ms per step).
    const int slots = decrypt_slots();
    auto fill = [&](int cols) {
        const double waves = (double)B * (double)((m + cols - 1) / cols) / slots;
        return waves / std::ceil(waves);
    };
    const bool narrow = slots > 0 && fill(256) > fill(512) + 0.1;
    const int cols = narrow ? 256 : 512;
    if ((m + cols - 1) / cols > 65535) return cudaErrorInvalidValue;
    const dim3 grid((unsigned)B, (m + cols - 1) / cols);
    if (narrow)
        k_decrypt<false, 4><<<grid, kDecThreads, smem, s>>>(PT, m, st, t_x, Nx, Yhat, Y, nullptr, vec);
    else
        k_decrypt<false, 2><<<grid, kDecThreads, smem, s>>>(PT, m, st, t_x, Nx, Yhat, Y, nullptr, vec);
    note_launch();
    return cudaGetLastError();
}

cudaError_t launch_check(const uint32_t *Xhat, int K, const uint32_t *Yhat, int m, const uint32_t *g,
                         const uint32_t *u, uint32_t ell, int B, int32_t *accept, cudaStream_t s) {
    if (B <= 0) return cudaSuccess;
    k_check<<<(unsigned)B, kCheckThreads, 0, s>>>(Xhat, K, Yhat, m, g, u, ell, accept); note_launch();
    return cudaGetLastError();
}

}  // namespace pv
