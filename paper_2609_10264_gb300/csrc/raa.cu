// RAA code kernels (App. B of the paper) and the sparse sampler.
//
//  * k_sample_sparse      draws e <- E_t^N (Sec. 3 notation) on the device.
//  * k_syndrome_scan      first half of the syndrome x' = G e for a sparse e:
//                         step function A e, permutation, and the suffix-sum
//                         accumulator as a single-pass decoupled look-back scan.
//  * k_syndrome_gather    second half: inverse permutation gather and the
//                         block sums of R, fused with x_hat = x + x'.
//  * k_encode_scan        one accumulate stage of the encoding G^T w over many
//                         lanes (preprocessing of P^T and Q, Sec. 6.3).
#include "common.cuh"
#include "launch.h"

namespace pv {
namespace {

__device__ __forceinline__ int bitlen32(uint32_t v) { return v ? 32 - __clz(v) : 0; }

// -----------------------------------------------------------------------------
// Sparse sampler: one warp per vector.  Specification (shared with the oracle,
// written independently there): the support is the first t distinct values of
// the sequence below(N) read from the ChaCha20 stream with nonce
// (tag, 2 idx); below(k) keeps the top bitlen(k-1) bits of a 32-bit word and
// rejects values >= k.  Values are the first t words of stream (tag, 2 idx + 1)
// whose top 31 bits lie in [1, q); the k-th one goes to the k-th smallest
// support index.
// -----------------------------------------------------------------------------
__global__ void __launch_bounds__(32) k_sample_sparse(pvmvmd_key key, uint32_t tag, uint64_t idx0,
                                                     uint32_t N, uint32_t t,
                                                     uint32_t *__restrict__ out,
                                                     unsigned long long *__restrict__ clear,
                                                     size_t clear_words) {
    extern __shared__ uint32_t sm[];
    const uint32_t nbw = (N + 31) / 32;
    uint32_t *bitmap = sm;
    uint32_t *words = sm + nbw;  // 512 keystream words = 32 blocks
    const int lane = threadIdx.x;

    for (size_t i = (size_t)blockIdx.x * 32 + lane; i < clear_words; i += (size_t)gridDim.x * 32)
        clear[i] = 0ull;

    const uint64_t idx = idx0 + blockIdx.x;
    uint32_t *supp = out + (size_t)blockIdx.x * 2 * t;
    uint32_t *vals = supp + t;
    for (uint32_t w = lane; w < nbw; w += 32) bitmap[w] = 0u;
    __syncwarp();

    // ---- support
    const uint64_t sidx = 2 * idx;
    uint32_t have = 0;
    if (N <= 1) {  // below(1) = 0 reads no word
        if (t >= 1 && lane == 0) bitmap[0] = 1u;
        have = t;
    }
    const int shift = 32 - (N > 1 ? bitlen32(N - 1) : 1);
    for (uint64_t wpos = 0; have < t; wpos += 512) {
        uint32_t blk[16];
        chacha20_block_dev(key, (uint32_t)(wpos / 16 + lane), tag, (uint32_t)sidx,
                           (uint32_t)(sidx >> 32), blk);
#pragma unroll
        for (int i = 0; i < 16; ++i) words[lane * 16 + i] = blk[i];
        __syncwarp();
        for (int batch = 0; batch < 16 && have < t; ++batch) {
            const uint32_t v = words[batch * 32 + lane] >> shift;
            const bool valid = v < N;
            const bool inset = valid && ((bitmap[v >> 5] >> (v & 31)) & 1u);
            const uint32_t vmask = __ballot_sync(kFull, valid);
            const uint32_t same = __match_any_sync(kFull, valid ? v : 0xffffffffu);
            const bool dup = (same & vmask & lanemask_lt()) != 0u;
            const bool cand = valid && !inset && !dup;
            const uint32_t cmask = __ballot_sync(kFull, cand);
            const uint32_t need = t - have;
            __syncwarp();  // every lane has read the bitmap before it changes
            if (cand && (uint32_t)__popc(cmask & lanemask_lt()) < need)
                atomicOr(&bitmap[v >> 5], 1u << (v & 31));
            have += min((uint32_t)__popc(cmask), need);
            __syncwarp();
        }
        __syncwarp();  // words are read before the next refill
    }

    // ---- ascending support from the bitmap
    uint32_t written = 0;
    for (uint32_t base = 0; base < nbw; base += 32) {
        uint32_t w = (base + lane < nbw) ? bitmap[base + lane] : 0u;
        const uint32_t c = __popc(w);
        uint32_t incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(kFull, incl, o);
            if (lane >= o) incl += y;
        }
        uint32_t pos = written + incl - c;
        while (w) {
            const int b = __ffs(w) - 1;
            supp[pos++] = (base + lane) * 32 + b;
            w &= w - 1;
        }
        written += __shfl_sync(kFull, incl, 31);
    }

    // ---- values in F*
    const uint64_t vidx = 2 * idx + 1;
    have = 0;
    for (uint64_t wpos = 0; have < t; wpos += 512) {
        uint32_t blk[16];
        chacha20_block_dev(key, (uint32_t)(wpos / 16 + lane), tag, (uint32_t)vidx,
                           (uint32_t)(vidx >> 32), blk);
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 16; ++i) words[lane * 16 + i] = blk[i];
        __syncwarp();
        for (int batch = 0; batch < 16 && have < t; ++batch) {
            const uint32_t v = words[batch * 32 + lane] >> 1;
            const bool valid = v != 0u && v < kQ;
            const uint32_t m = __ballot_sync(kFull, valid);
            const uint32_t r = __popc(m & lanemask_lt());
            if (valid && have + r < t) vals[have + r] = v;
            have = min(have + (uint32_t)__popc(m), t);
        }
    }
}

// -----------------------------------------------------------------------------
// Syndrome scan.  For sparse e with ascending support s_0 < ... < s_{t-1}:
//   (A e)_k = sum_{s_j >= k} e_j   (A_{i,j} = 1 iff i <= j: suffix sums)
//   c_i     = v2[pi2^-1(i)] * (A e)_{pi2^-1(i)}   ((Pi2 V2 A e)_i)
//   d       = A c                                 (suffix scan over i)
//   F_i     = v1_i * d_i                          ((V1 A Pi2 V2 A e)_i)
// Tiles of 2048 positions are processed from the end of the vector; each tile
// publishes its aggregate and then its inclusive suffix in one 64-bit status
// word (flag << 32 | value) and looks back over the tiles after it.
// -----------------------------------------------------------------------------
__global__ void __launch_bounds__(kScanThreads) k_syndrome_scan(
    const uint32_t *__restrict__ pi2inv, const uint32_t *__restrict__ v2p,
    const uint32_t *__restrict__ v1, uint32_t N, const uint32_t *__restrict__ sparse, uint32_t t,
    uint32_t count, uint32_t *__restrict__ F, unsigned long long *__restrict__ status,
    uint32_t *__restrict__ err) {
    extern __shared__ uint32_t sm[];
    uint32_t *s_supp = sm;     // t
    uint32_t *s_suf = sm + t;  // t + 1
    __shared__ uint32_t s_ticket, s_prefix, s_agg;
    __shared__ uint32_t s_wsum[kScanThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    if (tid == 0) s_ticket = atomicAdd(reinterpret_cast<unsigned int *>(status), 1u);
    __syncthreads();
    const uint32_t ntiles = scan_tiles(N);
    const uint32_t ticket = s_ticket;
    if (ticket >= count * ntiles) {  // status word not cleared: never index past the data
        if (tid == 0) record_error(err, kErrScanTimeout);
        return;
    }
    const uint32_t vec = ticket / ntiles;
    const uint32_t tile = ntiles - 1 - ticket % ntiles;
    unsigned long long *st = status + 1 + (size_t)vec * ntiles;

    const uint32_t *sp = sparse + (size_t)vec * 2 * t;
    for (uint32_t j = tid; j < t; j += kScanThreads) {
        s_supp[j] = sp[j];
        s_suf[j] = sp[t + j];
    }
    __syncthreads();
    if (warp == 0) {  // s_suf[j] <- sum_{j' >= j} e_{j'}; s_suf[t] = 0
        const uint32_t per = (t + 31) / 32;
        const uint32_t lo = min(t, lane * per), hi = min(t, lo + per);
        uint32_t sum = 0;
        for (uint32_t j = hi; j-- > lo;) sum = fadd(sum, s_suf[j]);
        uint32_t incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_down_sync(kFull, incl, o);
            if (lane + o < 32) incl = fadd(incl, y);
        }
        uint32_t run = fsub(incl, sum);
        for (uint32_t j = hi; j-- > lo;) {
            run = fadd(run, s_suf[j]);
            s_suf[j] = run;
        }
        if (lane == 0) s_suf[t] = 0;
    }
    __syncthreads();

    const uint32_t base = tile * kScanTile + tid * kScanItems;
    uint32_t c[kScanItems];
    uint32_t idx[kScanItems], scale[kScanItems];
    if (base + kScanItems <= N) {
        const uint4 a0 = *reinterpret_cast<const uint4 *>(pi2inv + base);
        const uint4 a1 = *reinterpret_cast<const uint4 *>(pi2inv + base + 4);
        const uint4 b0 = *reinterpret_cast<const uint4 *>(v2p + base);
        const uint4 b1 = *reinterpret_cast<const uint4 *>(v2p + base + 4);
        idx[0] = a0.x; idx[1] = a0.y; idx[2] = a0.z; idx[3] = a0.w;
        idx[4] = a1.x; idx[5] = a1.y; idx[6] = a1.z; idx[7] = a1.w;
        scale[0] = b0.x; scale[1] = b0.y; scale[2] = b0.z; scale[3] = b0.w;
        scale[4] = b1.x; scale[5] = b1.y; scale[6] = b1.z; scale[7] = b1.w;
    } else {
#pragma unroll
        for (int u = 0; u < kScanItems; ++u) {
            const uint32_t i = base + u;
            idx[u] = i < N ? pi2inv[i] : 0u;
            scale[u] = i < N ? v2p[i] : 0u;
        }
    }
#pragma unroll
    for (int u = 0; u < kScanItems; ++u) {
        uint32_t lo = 0, hi = t;  // first support index >= idx[u]
        while (lo < hi) {
            const uint32_t mid = (lo + hi) >> 1;
            if (s_supp[mid] < idx[u]) lo = mid + 1; else hi = mid;
        }
        c[u] = fmul(scale[u], s_suf[lo]);
    }
    uint32_t run = 0;
#pragma unroll
    for (int u = kScanItems - 1; u >= 0; --u) {
        run = fadd(run, c[u]);
        c[u] = run;
    }
    // block-wide exclusive suffix scan of the per-thread totals
    uint32_t incl = run;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_down_sync(kFull, incl, o);
        if (lane + o < 32) incl = fadd(incl, y);
    }
    if (lane == 0) s_wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        constexpr int nw = kScanThreads / 32;
        const uint32_t wv = lane < nw ? s_wsum[lane] : 0u;
        uint32_t winc = wv;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_down_sync(kFull, winc, o);
            if (lane + o < 32) winc = fadd(winc, y);
        }
        __syncwarp();
        if (lane < nw) s_wsum[lane] = fsub(winc, wv);
        if (lane == 0) s_agg = winc;
    }
    __syncthreads();
    const uint32_t thread_excl = fadd(fsub(incl, run), s_wsum[warp]);

    if (tid == 0) {
        const uint32_t agg = s_agg;
        uint32_t prefix = 0;
        if (tile == ntiles - 1) {
            st_release_u64(st + tile, (2ull << 32) | agg);
        } else {
            st_release_u64(st + tile, (1ull << 32) | agg);
            uint32_t j = tile + 1, spins = 0;
            for (;;) {
                const unsigned long long w = ld_acquire_u64(st + j);
                const uint32_t flag = (uint32_t)(w >> 32);
                if (flag == 0u) {
                    if (++spins > kSpinLimit) {
                        record_error(err, kErrScanTimeout);
                        break;
                    }
                    __nanosleep(32);
                    continue;
                }
                prefix = fadd(prefix, (uint32_t)w);
                if (flag == 2u || j + 1 >= ntiles) break;
                ++j;
            }
            st_release_u64(st + tile, (2ull << 32) | fadd(agg, prefix));
        }
        s_prefix = prefix;
    }
    __syncthreads();
    const uint32_t add = fadd(thread_excl, s_prefix);
    uint32_t *Fv = F + (size_t)vec * N;
#pragma unroll
    for (int u = 0; u < kScanItems; ++u) {
        const uint32_t i = base + u;
        if (i < N) Fv[i] = fmul(__ldg(v1 + i), fadd(c[u], add));
    }
}

// out_j = addend_j + sum_{c<r} F[pi1^-1(r j + c)]  ((R Pi1 F)_j, plus x_j).
__global__ void __launch_bounds__(256) k_syndrome_gather(const uint32_t *__restrict__ pi1inv,
                                                        uint32_t n, uint32_t r,
                                                        const uint32_t *__restrict__ F, uint32_t N,
                                                        const uint32_t *addend, uint32_t *out) {
    const uint32_t vec = blockIdx.y;
    const uint32_t j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= n) return;
    const uint32_t *Fv = F + (size_t)vec * N;
    const uint32_t *p = pi1inv + (size_t)j * r;
    uint32_t s = 0;
    if (r == 8) {
        const uint4 a = __ldg(reinterpret_cast<const uint4 *>(p));
        const uint4 b = __ldg(reinterpret_cast<const uint4 *>(p + 4));
        s = fadd(fadd(fadd(Fv[a.x], Fv[a.y]), fadd(Fv[a.z], Fv[a.w])),
                 fadd(fadd(Fv[b.x], Fv[b.y]), fadd(Fv[b.z], Fv[b.w])));
    } else {
        for (uint32_t c = 0; c < r; ++c) s = fadd(s, Fv[p[c]]);
    }
    const size_t o = (size_t)vec * n + j;
    out[o] = addend ? fadd(addend[o], s) : s;
}

// -----------------------------------------------------------------------------
// One accumulate stage of G^T w (App. B, encoding direction) over L lanes:
//   Y[j][l] = sum_{j' <= j} vscale[j'] * X[perm[j'] / div][l]
// With (perm, div, vscale) = (pi1, r, v1) this is A^T V1 Pi1^T R^T; with
// (pi2, 1, v2) it is A^T V2 Pi2^T.  A CTA owns 256 lanes and kEncTile
// positions; tiles of one lane block are chained by a decoupled look-back
// over per-lane aggregates (flags: 1 = aggregate, 2 = inclusive prefix).
// -----------------------------------------------------------------------------
template <bool kI8>
__global__ void __launch_bounds__(256) k_encode_scan(const void *__restrict__ Xv, size_t ldx,
                                                    const uint32_t *__restrict__ perm, uint32_t div,
                                                    const uint32_t *__restrict__ vscale, uint32_t N,
                                                    uint32_t L, uint32_t *__restrict__ Y, size_t ldy,
                                                    uint32_t *agg, uint32_t *incl, uint32_t *flags,
                                                    uint32_t *__restrict__ err) {
    __shared__ uint32_t s_ticket, s_flag;
    const int tid = threadIdx.x;
    const uint32_t nlb = (L + 255) / 256;
    const uint32_t ntiles = (N + kEncTile - 1) / kEncTile;
    if (tid == 0) s_ticket = atomicAdd(flags, 1u);
    __syncthreads();
    const uint32_t ticket = s_ticket;
    if (ticket >= nlb * ntiles) {  // flags not cleared: never index past the data
        if (tid == 0) record_error(err, kErrScanTimeout);
        return;
    }
    const uint32_t tile = ticket / nlb, lb = ticket % nlb;
    const uint32_t l = lb * 256 + tid;
    const bool lane_ok = l < L;
    const uint32_t j0 = tile * kEncTile;

    uint32_t v[kEncTile];
    uint32_t run = 0;
#pragma unroll
    for (int u = 0; u < kEncTile; ++u) {
        const uint32_t j = j0 + u;
        uint32_t x = 0;
        if (j < N && lane_ok) {
            const size_t src = __ldg(perm + j) / div;
            if (kI8)
                x = flift_i8(static_cast<const int8_t *>(Xv)[src * ldx + l]);
            else
                x = static_cast<const uint32_t *>(Xv)[src * ldx + l];
            x = fmul(__ldg(vscale + j), x);
        }
        run = fadd(run, x);
        v[u] = run;
    }

    const size_t slot = (size_t)lb * ntiles + tile;
    uint32_t *fl = flags + 1;
    uint32_t prefix = 0;
    if (tile == 0) {
        incl[slot * 256 + tid] = run;
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release_u32(fl + slot, 2u);
    } else {
        agg[slot * 256 + tid] = run;
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release_u32(fl + slot, 1u);
        for (uint32_t j = tile - 1;; --j) {
            const size_t ps = (size_t)lb * ntiles + j;
            if (tid == 0) {
                uint32_t f, spins = 0;
                while ((f = ld_acquire_u32(fl + ps)) == 0u) {
                    if (++spins > kSpinLimit) {
                        record_error(err, kErrScanTimeout);
                        f = 2u;
                        break;
                    }
                    __nanosleep(32);
                }
                s_flag = f;
            }
            __syncthreads();
            const uint32_t f = s_flag;
            prefix = fadd(prefix, f == 2u ? ld_cg_u32(incl + ps * 256 + tid)
                                          : ld_cg_u32(agg + ps * 256 + tid));
            __syncthreads();
            if (f == 2u || j == 0) break;
        }
        incl[slot * 256 + tid] = fadd(run, prefix);
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release_u32(fl + slot, 2u);
    }
    if (lane_ok) {
#pragma unroll
        for (int u = 0; u < kEncTile; ++u) {
            const uint32_t j = j0 + u;
            if (j < N) Y[j * ldy + l] = fadd(v[u], prefix);
        }
    }
}

__global__ void k_transpose_i8(const int8_t *__restrict__ in, int R, int C, int8_t *__restrict__ out) {
    __shared__ int8_t tile[32][33];
    const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int r = r0 + i, c = c0 + threadIdx.x;
        if (r < R && c < C) tile[i][threadIdx.x] = in[(size_t)r * C + c];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int c = c0 + i, r = r0 + threadIdx.x;
        if (r < R && c < C) out[(size_t)c * R + r] = tile[threadIdx.x][i];
    }
}

}  // namespace

// Bitmap of N bits plus 512 keystream words; covers N up to 8 * PVMVMD_MAX_K.
constexpr size_t kSampleMaxSmem = 200 * 1024;

cudaError_t launch_sample_sparse(const pvmvmd_key &key, uint32_t tag, uint64_t idx0, uint32_t N,
                                 uint32_t t, uint32_t count, uint32_t *out,
                                 unsigned long long *clear, size_t clear_words, cudaStream_t s) {
    if (count == 0) return cudaSuccess;
    const size_t smem = ((size_t)(N + 31) / 32 + 512) * sizeof(uint32_t);
    if (smem > kSampleMaxSmem) return cudaErrorInvalidValue;
    static const cudaError_t attr = cudaFuncSetAttribute(
        k_sample_sparse, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSampleMaxSmem);
    if (attr != cudaSuccess) return attr;
    k_sample_sparse<<<count, 32, smem, s>>>(key, tag, idx0, N, t, out, clear, clear_words);
    return cudaGetLastError();
}

cudaError_t launch_syndrome_scan(const uint32_t *pi2inv, const uint32_t *v2p, const uint32_t *v1,
                                 uint32_t N, const uint32_t *sparse, uint32_t t, uint32_t count,
                                 uint32_t *F, unsigned long long *status, uint32_t *err,
                                 cudaStream_t s) {
    if (count == 0) return cudaSuccess;
    const size_t smem = (2 * (size_t)t + 1) * sizeof(uint32_t);
    const unsigned grid = count * scan_tiles(N);
    k_syndrome_scan<<<grid, kScanThreads, smem, s>>>(pi2inv, v2p, v1, N, sparse, t, count, F, status,
                                                     err);
    return cudaGetLastError();
}

cudaError_t launch_syndrome_gather(const uint32_t *pi1inv, uint32_t n, uint32_t r,
                                   const uint32_t *F, uint32_t N, const uint32_t *addend,
                                   uint32_t *out, uint32_t count, cudaStream_t s) {
    if (count == 0 || n == 0) return cudaSuccess;
    dim3 grid((n + 255) / 256, count);
    k_syndrome_gather<<<grid, 256, 0, s>>>(pi1inv, n, r, F, N, addend, out);
    return cudaGetLastError();
}

size_t encode_scan_flag_words(uint32_t N, uint32_t L) {
    return 1 + (size_t)((L + 255) / 256) * ((N + kEncTile - 1) / kEncTile);
}
size_t encode_scan_value_words(uint32_t N, uint32_t L) {
    return (size_t)((L + 255) / 256) * ((N + kEncTile - 1) / kEncTile) * 256;
}

cudaError_t launch_encode_scan(const void *X, bool x_is_i8, size_t ldx, const uint32_t *perm,
                               uint32_t div, const uint32_t *vscale, uint32_t N, uint32_t L,
                               uint32_t *Y, size_t ldy, uint32_t *agg, uint32_t *incl,
                               uint32_t *flags, uint32_t *err, cudaStream_t s) {
    const size_t ctas = encode_scan_flag_words(N, L) - 1;
    if (ctas == 0) return cudaSuccess;
    if (ctas > 0x7fffffffu) return cudaErrorInvalidValue;
    if (x_is_i8)
        k_encode_scan<true><<<(unsigned)ctas, 256, 0, s>>>(X, ldx, perm, div, vscale, N, L, Y, ldy,
                                                           agg, incl, flags, err);
    else
        k_encode_scan<false><<<(unsigned)ctas, 256, 0, s>>>(X, ldx, perm, div, vscale, N, L, Y, ldy,
                                                            agg, incl, flags, err);
    return cudaGetLastError();
}

cudaError_t launch_transpose_i8(const int8_t *in, int R, int C, int8_t *out, cudaStream_t s) {
    if (R <= 0 || C <= 0) return cudaSuccess;
    dim3 grid((C + 31) / 32, (R + 31) / 32), block(32, 8);
    if (grid.y > 65535u) return cudaErrorInvalidValue;
    k_transpose_i8<<<grid, block, 0, s>>>(in, R, C, out);
    return cudaGetLastError();
}

}  // namespace pv
