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
//  * k_lane_*             the syndrome for a batch of vectors held as the lanes
//                         of an N x B array (sample, step function, scan, gather).
#include <map>
#include <mutex>
#include <cooperative_groups.h>

#include "common.cuh"
#include "launch.h"

namespace cg = cooperative_groups;

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
// Warp: mark the support of e <- E_t^N in `bitmap` (N bits, cleared by the
// caller) from stream (tag, sidx), using `words` (512 words) as keystream buffer.
__device__ void warp_sample_support(const pvmvmd_key &key, uint32_t tag, uint64_t sidx, uint32_t N,
                                    uint32_t t, uint32_t *bitmap, uint32_t *words, int lane) {
    uint32_t have = 0;
    if (N <= 1) {  // below(1) = 0 reads no word
        if (t >= 1 && lane == 0) bitmap[0] = 1u;
        __syncwarp();
        return;
    }
    const int shift = 32 - bitlen32(N - 1);
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
}

// Warp: as warp_sample_support, and also writes the accepted indices, in the
// order they were accepted, to list[0..t).
__device__ void warp_sample_support_list(const pvmvmd_key &key, uint32_t tag, uint64_t sidx,
                                         uint32_t N, uint32_t t, uint32_t *bitmap, uint32_t *words,
                                         uint32_t *list, int lane) {
    uint32_t have = 0;
    if (N <= 1) {
        if (t >= 1 && lane == 0) list[0] = 0u;
        __syncwarp();
        return;
    }
    const int shift = 32 - bitlen32(N - 1);
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
            const uint32_t rk = __popc(cmask & lanemask_lt());
            __syncwarp();
            if (cand && rk < need) {
                atomicOr(&bitmap[v >> 5], 1u << (v & 31));
                list[have + rk] = v;
            }
            have += min((uint32_t)__popc(cmask), need);
            __syncwarp();
        }
        __syncwarp();
    }
}

// Warp: the set bits of `bitmap` (nbw words) in ascending order -> dst.
__device__ void warp_bitmap_to_support(const uint32_t *bitmap, uint32_t nbw, uint32_t *dst, int lane) {
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
            dst[pos++] = (base + lane) * 32 + b;
            w &= w - 1;
        }
        written += __shfl_sync(kFull, incl, 31);
    }
}

// Warp: the first t draws of F* from stream (tag, vidx) -> dst.
__device__ void warp_sample_values(const pvmvmd_key &key, uint32_t tag, uint64_t vidx, uint32_t t,
                                   uint32_t *words, uint32_t *dst, int lane) {
    uint32_t have = 0;
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
            if (valid && have + r < t) dst[have + r] = v;
            have = min(have + (uint32_t)__popc(m), t);
        }
    }
    __syncwarp();
}

// One warp per vector (the path for codes too long for one cluster).
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
    for (uint32_t w = lane; w < nbw; w += 32) bitmap[w] = 0u;
    __syncwarp();
    warp_sample_support(key, tag, 2 * idx, N, t, bitmap, words, lane);
    warp_bitmap_to_support(bitmap, nbw, supp, lane);
    warp_sample_values(key, tag, 2 * idx + 1, t, words, supp + t, lane);
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
    uint32_t *__restrict__ err, uint32_t skip_tile, uint32_t spin_limit) {
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
        // a failure-path test withholds this tile's status words, so that the
        // look-back of the tile before it expires (off: skip_tile >= ntiles)
        const bool publish = tile != skip_tile;
        uint32_t prefix = 0;
        if (tile == ntiles - 1) {
            if (publish) st_release_u64(st + tile, (2ull << 32) | agg);
        } else {
            if (publish) st_release_u64(st + tile, (1ull << 32) | agg);
            uint32_t j = tile + 1, spins = 0;
            for (;;) {
                const unsigned long long w = ld_acquire_u64(st + j);
                const uint32_t flag = (uint32_t)(w >> 32);
                if (flag == 0u) {
                    if (++spins > spin_limit) {
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
            if (publish) st_release_u64(st + tile, (2ull << 32) | fadd(agg, prefix));
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
// Fused syndrome: x' = G e for a freshly sampled sparse e, in one kernel per
// vector, with the length-N intermediate held in shared memory: one CTA of
// 1024 threads when it fits, else a thread-block cluster whose CTAs each hold
// a slice (CTA `rank` owns positions [rank*slice, (rank+1)*slice)) and read
// each other's through DSMEM.  Steps (App. B, syndrome direction):
//   sample e (warp 0: support; warp 1: values; every CTA of a cluster draws
//     the same keystream, rank 0 writes the state), the ascending support
//     read off the sampling bitmap by a block-wide scan;
//   c_i = v2[pi2^-1(i)] * (A e)_{pi2^-1(i)}, the step function (A e)_k found
//     through a bucket index over the sorted support;
//   d = A c: a block suffix scan plus the aggregates of later CTAs;
//   F_i = v1_i * d_i;  out_j = addend_j + sum_{c<r} F[pi1^-1(r j + c)].
// No global scratch and no look-back.
// -----------------------------------------------------------------------------
constexpr int kFusedThreads = 1024;
constexpr int kFusedBuckets = 512;   // index over the sorted support
constexpr int kFusedBatch = 16;      // loads in flight per thread
constexpr int kFusedBatch1 = 8;      // the same in the single-CTA scatter

__device__ __forceinline__ uint32_t fpad(uint32_t i) { return i + (i >> 5); }  // bank padding

// floor(x / d) as (x * ceil(2^40 / d)) >> 40 (division by an invariant
// integer through a rounded-up reciprocal, Granlund and Montgomery 1994).
// Exact when x * d < 2^40: the product is x / d + x * eps / 2^40 with
// 0 <= eps < 1, and x / 2^40 < 1 / d never reaches the next integer.
__host__ __device__ __forceinline__ uint64_t div_magic(uint32_t d) { return ((1ull << 40) + d - 1) / d; }
__device__ __forceinline__ uint32_t div_by(uint32_t x, uint64_t magic) {
    return (uint32_t)(((uint64_t)x * magic) >> 40);
}

// Everything before this point reads only the key and the code tables; the
// state st and the output are written after griddepcontrol.wait, so a launch
// with programmatic serialisation may run its sampling and scans while the
// kernel before it finishes.  Writes st = (support, e) with e_j recovered
// from the suffix sums suf (suf[t] = 0).
__device__ __forceinline__ void fused_publish(uint32_t *st, const uint32_t *supp, const uint32_t *suf,
                                              uint32_t t, int tid) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    for (uint32_t j = tid; j < t; j += kFusedThreads) {
        st[j] = supp[j];
        st[t + j] = fsub(suf[j], suf[j + 1]);
    }
}

__global__ void __launch_bounds__(kFusedThreads) k_syndrome_fused(
    pvmvmd_key key, uint32_t tag, uint64_t idx0, uint32_t N, uint32_t t, uint32_t slice,
    const uint32_t *__restrict__ pi2inv, const uint32_t *__restrict__ v2p,
    const uint32_t *__restrict__ v1, const uint32_t *__restrict__ pi1inv, uint32_t n, uint32_t r,
    uint32_t *__restrict__ sparse_out, const uint32_t *addend, uint32_t *out,
    const uint32_t *__restrict__ pi2, const uint32_t *__restrict__ v2m,
    const uint32_t *__restrict__ v1pm) {
    cg::cluster_group cluster = cg::this_cluster();
    extern __shared__ uint32_t sm[];
    __shared__ uint32_t s_wsum[kFusedThreads / 32];
    __shared__ uint32_t s_texcl[kFusedThreads];
    __shared__ uint32_t s_first[kFusedBuckets];
    __shared__ uint32_t s_agg;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t C = cluster.num_blocks(), rank = cluster.block_rank();
    const uint32_t vec = blockIdx.y;
    const uint64_t idx = idx0 + vec;
    const uint32_t fwords = fpad(slice);
    uint32_t *F = sm;                 // padded slice (bitmap while sampling)
    uint32_t *supp = sm + fwords;     // t
    uint32_t *suf = supp + t;         // t + 1
    uint32_t *words0 = suf + t + 1;   // 512
    uint32_t *words1 = words0 + 512;  // 512 (then the unsorted support list)
    uint32_t *list = words1 + 512;    // t
    const uint32_t nbw = (N + 31) / 32;

    // the kernels that follow may launch now; they wait for this one before
    // reading anything it writes
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    // ---- sample e: warp 0 the support, warp 1 the values
    for (uint32_t w = tid; w < nbw; w += kFusedThreads) F[w] = 0u;
    __syncthreads();
    if (warp == 0)
        warp_sample_support_list(key, tag, 2 * idx, N, t, F, words0, list, lane);
    else if (warp == 1)
        warp_sample_values(key, tag, 2 * idx + 1, t, words1, suf, lane);
    __syncthreads();
    {
        // ascending support: the set bits of the sampling bitmap, compacted
        // with a block-wide exclusive scan of the per-thread bit counts
        const uint32_t per = (nbw + kFusedThreads - 1) / kFusedThreads;
        const uint32_t w0 = min(nbw, tid * per), w1 = min(nbw, w0 + per);
        uint32_t cnt = 0;
        for (uint32_t w = w0; w < w1; ++w) cnt += __popc(F[w]);
        uint32_t incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(kFull, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) s_wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            constexpr int nw = kFusedThreads / 32;
            const uint32_t wv = lane < nw ? s_wsum[lane] : 0u;
            uint32_t wi = wv;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_up_sync(kFull, wi, o);
                if (lane >= o) wi += y;
            }
            __syncwarp();
            if (lane < nw) s_wsum[lane] = wi - wv;
        }
        __syncthreads();
        uint32_t pos = s_wsum[warp] + incl - cnt;
        for (uint32_t w = w0; w < w1; ++w) {
            uint32_t bits = F[w];
            while (bits) {
                supp[pos++] = w * 32 + (uint32_t)(__ffs(bits) - 1);
                bits &= bits - 1;
            }
        }
    }
    __syncthreads();
    if (warp == 0) {  // suf[j] <- sum_{j' >= j} e_{j'}; suf[t] = 0
        const uint32_t per = (t + 31) / 32;
        const uint32_t lo = min(t, lane * per), hi = min(t, lo + per);
        uint32_t sum = 0;
        for (uint32_t j = hi; j-- > lo;) sum = fadd(sum, suf[j]);
        uint32_t incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_down_sync(kFull, incl, o);
            if (lane + o < 32) incl = fadd(incl, y);
        }
        uint32_t run = fsub(incl, sum);
        for (uint32_t j = hi; j-- > lo;) {
            run = fadd(run, suf[j]);
            suf[j] = run;
        }
        if (lane == 0) suf[t] = 0;
    }
    if (C == 1) {
        // ---- the whole vector in this CTA: c_{pi2(k)} = v2_k (A e)_k,
        // scattered into the slice.  Positions are interleaved over the
        // threads (k = u * 1024 + tid), so the table loads are coalesced and
        // kFusedBatch1 of them are in flight per thread; (A e)_k is found
        // from a bucket index into the sorted support.
        int bshift = 0;
        while ((N >> bshift) > (uint32_t)kFusedBuckets - 1) ++bshift;
        const uint32_t nbk = (N >> bshift) + 1;
        for (uint32_t b = tid; b < nbk; b += kFusedThreads) {
            const uint32_t start = b << bshift;
            uint32_t lo = 0, hi = t;
            while (lo < hi) {
                const uint32_t mid = (lo + hi) >> 1;
                if (supp[mid] < start) lo = mid + 1; else hi = mid;
            }
            s_first[b] = lo;
        }
        __syncthreads();
        const uint32_t items = slice / kFusedThreads;
        for (uint32_t i = N + tid; i < slice; i += kFusedThreads) F[fpad(i)] = 0u;  // padding
        for (uint32_t u0 = 0; u0 < items; u0 += kFusedBatch1) {
            uint32_t pk[kFusedBatch1], vk[kFusedBatch1];
#pragma unroll
            for (int u = 0; u < kFusedBatch1; ++u) {
                const uint32_t k = (u0 + u) * kFusedThreads + tid;
                const bool ok = u0 + u < items && k < N;
                pk[u] = ok ? __ldg(pi2 + k) : 0u;
                vk[u] = ok ? __ldg(v2m + k) : 0u;
            }
#pragma unroll
            for (int u = 0; u < kFusedBatch1; ++u) {
                const uint32_t k = (u0 + u) * kFusedThreads + tid;
                if (u0 + u < items && k < N) {
                    uint32_t j = s_first[k >> bshift];
                    while (j < t && supp[j] < k) ++j;
                    F[fpad(pk[u])] = fmul_mont(suf[j], vk[u]);
                }
            }
        }
        __syncthreads();
        // d = A c: thread tid owns positions [tid*items, (tid+1)*items)
        uint32_t run = 0;
        for (uint32_t u = items; u-- > 0;) {
            const uint32_t li = tid * items + u;
            run = fadd(run, F[fpad(li)]);
            F[fpad(li)] = run;
        }
        uint32_t incl = run;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_down_sync(kFull, incl, o);
            if (lane + o < 32) incl = fadd(incl, y);
        }
        if (lane == 0) s_wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            constexpr int nw = kFusedThreads / 32;
            const uint32_t wv = lane < nw ? s_wsum[lane] : 0u;
            uint32_t winc = wv;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_down_sync(kFull, winc, o);
                if (lane + o < 32) winc = fadd(winc, y);
            }
            __syncwarp();
            if (lane < nw) s_wsum[lane] = fsub(winc, wv);
        }
        __syncthreads();
        const uint32_t add = fadd(fsub(incl, run), s_wsum[warp]);
        for (uint32_t u = 0; u < items; ++u) {
            const uint32_t li = tid * items + u;
            F[fpad(li)] = fadd(F[fpad(li)], add);
        }
        __syncthreads();
        fused_publish(sparse_out + (size_t)vec * 2 * t, supp, suf, t, tid);
        // out_j = addend_j + sum_c v1[pi1^-1(r j + c)] d[pi1^-1(r j + c)]
        for (uint32_t jo = tid; jo < n; jo += kFusedThreads) {
            const uint32_t *p = pi1inv + (size_t)jo * r;
            const uint32_t *w = v1pm + (size_t)jo * r;
            uint32_t acc = 0;
            if (r == 8) {
                const uint4 a = __ldg(reinterpret_cast<const uint4 *>(p));
                const uint4 b = __ldg(reinterpret_cast<const uint4 *>(p + 4));
                const uint4 c = __ldg(reinterpret_cast<const uint4 *>(w));
                const uint4 d = __ldg(reinterpret_cast<const uint4 *>(w + 4));
                acc = fadd(fadd(fadd(fmul_mont(F[fpad(a.x)], c.x), fmul_mont(F[fpad(a.y)], c.y)),
                                fadd(fmul_mont(F[fpad(a.z)], c.z), fmul_mont(F[fpad(a.w)], c.w))),
                           fadd(fadd(fmul_mont(F[fpad(b.x)], d.x), fmul_mont(F[fpad(b.y)], d.y)),
                                fadd(fmul_mont(F[fpad(b.z)], d.z), fmul_mont(F[fpad(b.w)], d.w))));
            } else {
                for (uint32_t cc = 0; cc < r; ++cc) acc = fadd(acc, fmul_mont(F[fpad(__ldg(p + cc))], __ldg(w + cc)));
            }
            const size_t o = (size_t)vec * n + jo;
            out[o] = addend ? fadd(addend[o], acc) : acc;
        }
        return;
    }

    // bucket index: position k lies in bucket k >> bshift; s_first[b] is the
    // first support index >= b << bshift
    int bshift = 0;
    while ((N >> bshift) > (uint32_t)kFusedBuckets - 1) ++bshift;
    const uint32_t nbk = (N >> bshift) + 1;
    for (uint32_t b = tid; b < nbk; b += kFusedThreads) {
        const uint32_t start = b << bshift;
        uint32_t lo = 0, hi = t;
        while (lo < hi) {
            const uint32_t mid = (lo + hi) >> 1;
            if (supp[mid] < start) lo = mid + 1; else hi = mid;
        }
        s_first[b] = lo;
    }
    __syncthreads();

    // ---- c over this CTA's slice (coalesced positions, loads batched)
    const uint32_t base = rank * slice;
    const uint32_t items = slice / kFusedThreads;
    const uint64_t items_magic = div_magic(items), slice_magic = div_magic(slice);
    for (uint32_t u0 = 0; u0 < items; u0 += kFusedBatch) {
        uint32_t kk[kFusedBatch], sc[kFusedBatch];
#pragma unroll
        for (int u = 0; u < kFusedBatch; ++u) {
            const uint32_t i = base + (u0 + u) * kFusedThreads + tid;
            const bool ok = u0 + u < items && i < N;
            kk[u] = ok ? __ldg(pi2inv + i) : 0u;
            sc[u] = ok ? __ldg(v2p + i) : 0u;
        }
#pragma unroll
        for (int u = 0; u < kFusedBatch; ++u) {
            if (u0 + u < items) {
                uint32_t j = s_first[kk[u] >> bshift];  // first support index >= kk[u]
                while (j < t && supp[j] < kk[u]) ++j;
                F[fpad((u0 + u) * kFusedThreads + tid)] = fmul(sc[u], suf[j]);
            }
        }
    }
    __syncthreads();
    // ---- suffix sums: thread tid owns [tid*items, (tid+1)*items)
    uint32_t run = 0;
    for (uint32_t u = items; u-- > 0;) {
        const uint32_t li = tid * items + u;
        run = fadd(run, F[fpad(li)]);
        F[fpad(li)] = run;
    }
    uint32_t incl = run;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_down_sync(kFull, incl, o);
        if (lane + o < 32) incl = fadd(incl, y);
    }
    if (lane == 0) s_wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        constexpr int nw = kFusedThreads / 32;
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
    s_texcl[tid] = fadd(fsub(incl, run), s_wsum[warp]);
    uint32_t after = 0;  // sum over the positions owned by later CTAs
    if (C > 1) {
        cluster.sync();
        // every warp reads the later ranks' totals at once (one DSMEM load
        // per lane) and sums them with shuffles
        const uint32_t rr = rank + 1 + (uint32_t)lane;
        after = rr < C ? *cluster.map_shared_rank(&s_agg, rr) : 0u;
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) after = fadd(after, __shfl_xor_sync(kFull, after, o));
    } else {
        __syncthreads();
    }
    for (uint32_t u0 = 0; u0 < items; u0 += kFusedBatch) {
        uint32_t sc[kFusedBatch];
#pragma unroll
        for (int u = 0; u < kFusedBatch; ++u) {
            const uint32_t i = base + (u0 + u) * kFusedThreads + tid;
            sc[u] = (u0 + u < items && i < N) ? __ldg(v1 + i) : 0u;
        }
#pragma unroll
        for (int u = 0; u < kFusedBatch; ++u) {
            if (u0 + u < items) {
                const uint32_t li = (u0 + u) * kFusedThreads + tid;
                const uint32_t d = fadd(F[fpad(li)], fadd(s_texcl[div_by(li, items_magic)], after));
                F[fpad(li)] = fmul(sc[u], d);
            }
        }
    }
    if (C > 1) cluster.sync(); else __syncthreads();
    if (rank == 0) fused_publish(sparse_out + (size_t)vec * 2 * t, supp, suf, t, tid);
    else asm volatile("griddepcontrol.wait;" ::: "memory");

    // ---- gather: out_j = addend_j + sum_c F[pi1^-1(r j + c)]
    const uint32_t nsl = (n + C - 1) / C;
    const uint32_t j0 = rank * nsl, j1 = min(n, j0 + nsl);
    for (uint32_t j = j0 + tid; j < j1; j += kFusedThreads) {
        const uint32_t *p = pi1inv + (size_t)j * r;
        uint32_t acc = 0;
        if (r == 8) {
            const uint4 a = __ldg(reinterpret_cast<const uint4 *>(p));
            const uint4 b = __ldg(reinterpret_cast<const uint4 *>(p + 4));
            const uint32_t gi[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
            uint32_t v[8];
            if (C == 1) {
#pragma unroll
                for (int c = 0; c < 8; ++c) v[c] = F[fpad(gi[c])];
            } else {
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const uint32_t owner = div_by(gi[c], slice_magic);
                    v[c] = cluster.map_shared_rank(F, owner)[fpad(gi[c] - owner * slice)];
                }
            }
#pragma unroll
            for (int c = 0; c < 8; ++c) acc = fadd(acc, v[c]);
        } else {
            for (uint32_t c = 0; c < r; ++c) {
                const uint32_t gi = __ldg(p + c);
                const uint32_t owner = div_by(gi, slice_magic), off = gi - owner * slice;
                acc = fadd(acc, C == 1 ? F[fpad(off)] : cluster.map_shared_rank(F, owner)[fpad(off)]);
            }
        }
        const size_t o = (size_t)vec * n + j;
        out[o] = addend ? fadd(addend[o], acc) : acc;
    }
    if (C > 1) cluster.sync();  // peers may still read this CTA's F
}

// -----------------------------------------------------------------------------
// One accumulate stage of G^T w (App. B, encoding direction) over L lanes:
//   Y[j][l] = sum_{j' <= j} vscale[j'] * X[perm[j'] / div][l]
// With (perm, div, vscale) = (pi1, r, v1) this is A^T V1 Pi1^T R^T; with
// (pi2, 1, v2) it is A^T V2 Pi2^T.  vscale_m holds vscale in Montgomery form
// (v R mod q).  A CTA owns 256 lanes and kEncTile positions: the source row
// and scale of each position are looked up once per CTA (in shared memory),
// and every thread issues all kEncTile row loads of its lane before the
// arithmetic.  Tiles of one lane block are chained by a decoupled look-back
// that each lane walks on its own: per (tile, lane) one 64-bit status word
// holds a state in its high half (1: the tile's own sum, 2: the inclusive
// prefix through the tile) and the value in its low half, so a reader gets
// state and value in one load and no fence or block barrier is needed.
// Tiles are numbered in the order CTAs start (a global ticket), so every
// predecessor of a tile is already running.  (The earlier form, one flag per
// tile and the lanes' values in separate arrays behind a fence and block
// barriers, with warp 0 reading 32 flags at a time, took 0.755 ms per
// 4096 x 4096 encoding.)  At 32 positions per tile the kernel is held to 64
// registers, four CTAs per SM.
// -----------------------------------------------------------------------------
__device__ __forceinline__ unsigned long long enc_status(uint32_t state, uint32_t v) {
    return ((unsigned long long)state << 32) | v;
}

template <bool kI8>
__global__ void __launch_bounds__(256, 4) k_encode_scan(const void *__restrict__ Xv, size_t ldx,
                                                    const uint32_t *__restrict__ perm, uint32_t div,
                                                    const uint32_t *__restrict__ vscale_m, uint32_t N,
                                                    uint32_t L, uint32_t *__restrict__ Y, size_t ldy,
                                                    unsigned long long *status, uint32_t *ticket_ctr,
                                                    uint32_t *__restrict__ err) {
    __shared__ uint32_t s_ticket;
    __shared__ unsigned long long s_off[kEncTile];  // source row offset (row * ldx) of each position
    __shared__ uint32_t s_vs[kEncTile];
    const int tid = threadIdx.x;
    const uint32_t nlb = (L + 255) / 256;
    const uint32_t ntiles = (N + kEncTile - 1) / kEncTile;
    if (tid == 0) s_ticket = atomicAdd(ticket_ctr, 1u);
    __syncthreads();
    const uint32_t ticket = s_ticket;
    if (ticket >= nlb * ntiles) {  // ticket not cleared: never index past the data
        if (tid == 0) record_error(err, kErrScanTimeout);
        return;
    }
    const uint32_t tile = ticket / nlb, lb = ticket % nlb;
    const uint32_t l = lb * 256 + tid;
    const bool lane_ok = l < L;
    const uint32_t j0 = tile * kEncTile;
    if (tid < kEncTile) {
        const uint32_t j = j0 + tid;
        s_off[tid] = (unsigned long long)(j < N ? __ldg(perm + j) / div : 0u) * ldx;
        s_vs[tid] = j < N ? __ldg(vscale_m + j) : 0u;  // 0 past N: adds nothing
    }
    __syncthreads();

    uint32_t v[kEncTile];
#pragma unroll
    for (int u = 0; u < kEncTile; ++u) {
        const bool ok = lane_ok && j0 + u < N;
        const size_t src = (size_t)s_off[u] + l;
        if (kI8)
            v[u] = ok ? flift_i8(static_cast<const int8_t *>(Xv)[src]) : 0u;
        else
            v[u] = ok ? static_cast<const uint32_t *>(Xv)[src] : 0u;
    }
    uint32_t run = 0;
#pragma unroll
    for (int u = 0; u < kEncTile; ++u) {
        run = fadd(run, fmul_mont(v[u], s_vs[u]));
        v[u] = run;
    }

    // this lane's status word of tile 0 of the lane block; tile p is p * 256 on
    unsigned long long *sw = status + (size_t)lb * ntiles * 256 + tid;
    uint32_t prefix = 0;
    if (tile == 0) {
        st_relaxed_u64(sw, enc_status(2u, run));
    } else {
        st_relaxed_u64(sw + (size_t)tile * 256, enc_status(1u, run));
        uint32_t spins = 0;
        for (uint32_t p = tile - 1;;) {
            const unsigned long long w = ld_relaxed_u64(sw + (size_t)p * 256);
            const uint32_t state = (uint32_t)(w >> 32);
            if (state == 0u) {
                if (++spins > kSpinLimit) {
                    record_error(err, kErrScanTimeout);
                    break;
                }
                __nanosleep(32);
                continue;
            }
            prefix = fadd(prefix, (uint32_t)w);
            if (state == 2u || p == 0u) break;  // tile 0 is always inclusive
            --p;
        }
        st_relaxed_u64(sw + (size_t)tile * 256, enc_status(2u, fadd(run, prefix)));
    }
    if (lane_ok) {
        uint32_t *yp = Y + (size_t)j0 * ldy + l;
        const uint32_t nu = N - j0 < (uint32_t)kEncTile ? N - j0 : (uint32_t)kEncTile;
#pragma unroll
        for (int u = 0; u < kEncTile; ++u, yp += ldy)
            if ((uint32_t)u < nu) *yp = fadd(v[u], prefix);
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

// -----------------------------------------------------------------------------
// Lane-parallel syndrome x' = G e for a batch of L vectors (Encrypt at large
// batch).  The vectors are the lanes of an N x Lp array C (Lp = L rounded up
// to a multiple of 4, lane index contiguous), so every permutation step of
// G = R Pi1 V1 A Pi2 V2 A moves whole rows:
//   C[pi2(k)][b] = v2_k (A e_b)_k,  (A e_b)_k = sum_{j: s_j >= k} e_j
//                                                   (k_lane_expand)
//   agg[tau][b]  = sum of C[i][b] over tile tau     (k_lane_tile_sum)
//   carry[tau][b] = sum_{tau' > tau} agg[tau'][b]   (k_lane_carry)
//   C[i][b] <- v1_i (carry + sum_{i' >= i in the tile} C[i'][b])
//                                                   (k_lane_scan, in place)
//   out[b][j] = addend[b][j] + sum_{c<r} C[pi1^-1(r j + c)][b]
//                                                   (k_lane_gather)
// A thread owns four consecutive lanes (16-byte accesses) of one tile or
// span; a CTA of 256 threads covers `cols` lane quads (Lp/4 rounded up to a
// power of two, at most 64) of 256 / cols tiles or spans.  The six kernels launch with
// programmatic serialisation and wait (griddepcontrol.wait) before touching
// their predecessor's output.  Only the sampler, whose work needs the key
// alone, lets its successor launch early; the others let it launch at their
// completion.  Early launches of the large grids held SM slots with waiting
// CTAs and were slower (K = 28672, B = 256: 341 against 307 us).
// -----------------------------------------------------------------------------
constexpr int kLaneTileMin = 32;   // positions per tile (one thread walks them):
constexpr int kLaneTileMax = 128;  // the launch picks 32, 64 or 128
constexpr int kLaneCta = 256;      // threads per lane CTA
constexpr int kLaneQuadsMax = 64;  // lane quads per CTA (256 lanes)
constexpr int kExpandSpan = 16;    // positions per expand thread (a multiple of 4)
constexpr int kLaneBuckets = 256;  // bucket index into each lane's sorted support
constexpr int kGatherJ = 16;       // outputs per gather CTA
constexpr int kCarryThreads = 1024;  // tile chunks per lane quad in the carry kernel

__host__ __device__ inline uint32_t lane_pad(uint32_t L) { return (L + 3) & ~3u; }
// Lane quads per CTA: Lp/4 rounded up to a power of two, at most 64 (a CTA
// then holds 256 / cols tiles or spans, and no thread idles for Lp/4 = 16).
__host__ __device__ inline uint32_t lane_cols(uint32_t L) {
    const uint32_t q = lane_pad(L) / 4;
    uint32_t c = 1;
    while (c < q && c < (uint32_t)kLaneQuadsMax) c *= 2;
    return c;
}
__device__ __forceinline__ uint4 fadd4(uint4 a, uint4 b) {
    return make_uint4(fadd(a.x, b.x), fadd(a.y, b.y), fadd(a.z, b.z), fadd(a.w, b.w));
}

// Positions q << lane_bshift(N), q < kLaneBuckets, cover [0, N).
__host__ __device__ inline uint32_t lane_bshift(uint32_t N) {
    uint32_t b = 0;
    while (b < 31 && ((N - 1) >> b) >= (uint32_t)kLaneBuckets) ++b;
    return N > 1 ? b : 0u;
}

// e_b for vector idx0 + blockIdx.x as in k_sample_sparse (warp 0 the
// support, warp 1 the values), written as st[b] = (ascending support,
// values), S[b][j] = sum_{j' >= j} values[j'], S[b][t] = 0, and the bucket
// index first[b][q] = the first support index at or above position
// q << lane_bshift(N).  Everything is computed in shared memory from the key
// alone; st, S and first are written after griddepcontrol.wait (a kernel
// before this one may still read them).
__global__ void __launch_bounds__(128) k_lane_sample(pvmvmd_key key, uint32_t tag, uint64_t idx0,
                                                    uint32_t N, uint32_t t, uint32_t *__restrict__ st,
                                                    uint32_t *__restrict__ S, uint16_t *__restrict__ first) {
    extern __shared__ uint32_t sm[];
    const uint32_t nbw = (N + 31) / 32;
    uint32_t *bitmap = sm;
    uint32_t *words = sm + nbw;      // 512 keystream words (support)
    uint32_t *words2 = words + 512;  // 512 keystream words (values)
    uint32_t *list = words2 + 512;   // t, in the order accepted
    uint32_t *vals = list + t;       // t
    uint32_t *sorted = vals + t;     // t
    uint32_t *suf = sorted + t;      // t + 1
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const uint64_t idx = idx0 + blockIdx.x;
    for (uint32_t w = tid; w < nbw; w += 128) bitmap[w] = 0u;
    __syncthreads();
    if (warp == 0) warp_sample_support_list(key, tag, 2 * idx, N, t, bitmap, words, list, lane);
    else if (warp == 1) warp_sample_values(key, tag, 2 * idx + 1, t, words2, vals, lane);
    __syncthreads();
    for (uint32_t i = tid; i < t; i += 128) {  // ascending support by rank (entries distinct)
        const uint32_t v = list[i];
        uint32_t rk = 0;
        for (uint32_t j = 0; j < t; ++j) rk += list[j] < v;
        sorted[rk] = v;
    }
    if (warp == 0) {
        // suffix sums: lane owns a contiguous chunk, chunks combined by shuffles
        const uint32_t per = (t + 31) / 32;
        const uint32_t lo = min(t, lane * per), hi = min(t, lo + per);
        uint32_t sum = 0;
        for (uint32_t j = hi; j-- > lo;) sum = fadd(sum, vals[j]);
        uint32_t incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_down_sync(kFull, incl, o);
            if (lane + o < 32) incl = fadd(incl, y);
        }
        uint32_t run = fsub(incl, sum);  // sum over the chunks after this lane's
        for (uint32_t j = hi; j-- > lo;) {
            run = fadd(run, vals[j]);
            suf[j] = run;
        }
        if (lane == 0) suf[t] = 0u;
    }
    __syncthreads();
    const uint32_t bshift = lane_bshift(N);
    uint16_t fq[kLaneBuckets / 128];
#pragma unroll
    for (int h = 0; h < kLaneBuckets / 128; ++h) {
        const uint32_t pos = (uint32_t)(tid + 128 * h) << bshift;
        uint32_t lo = 0, hi = t;
        while (lo < hi) {
            const uint32_t mid = (lo + hi) >> 1;
            if (sorted[mid] < pos) lo = mid + 1; else hi = mid;
        }
        fq[h] = (uint16_t)lo;
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");
    uint32_t *stb = st + (size_t)blockIdx.x * 2 * t;
    uint32_t *Sb = S + (size_t)blockIdx.x * (t + 1);
    for (uint32_t j = tid; j < t; j += 128) {
        stb[j] = sorted[j];
        stb[t + j] = vals[j];
    }
    for (uint32_t j = tid; j <= t; j += 128) Sb[j] = suf[j];
#pragma unroll
    for (int h = 0; h < kLaneBuckets / 128; ++h)
        first[(size_t)blockIdx.x * kLaneBuckets + tid + 128 * h] = fq[h];
}

// C[pi2(k)][b] = v2_k (A e_b)_k: a thread walks kExpandSpan positions k of
// four lanes in order with a pointer per lane into the sorted support, and
// writes the four lanes of row pi2(k) with one 16-byte store.
__global__ void __launch_bounds__(kLaneCta) k_lane_expand(const uint32_t *__restrict__ st,
                                                         const uint32_t *__restrict__ S,
                                                         const uint16_t *__restrict__ first, uint32_t t,
                                                         uint32_t N, uint32_t L,
                                                         const uint32_t *__restrict__ pi2,
                                                         const uint32_t *__restrict__ v2m,
                                                         uint4 *__restrict__ C) {
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs come from the kernel before
    const uint32_t cols = lane_cols(L), Lq = lane_pad(L) / 4;
    const uint32_t g = blockIdx.y * cols + threadIdx.x % cols;
    const uint32_t k0 = (blockIdx.x * (kLaneCta / cols) + threadIdx.x / cols) * kExpandSpan;
    const uint32_t k1 = min(N, k0 + kExpandSpan);
    if (g >= Lq || k0 >= k1) return;
    uint32_t j[4], next[4], cur[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint32_t b = 4 * g + q;
        next[q] = 0xffffffffu;
        cur[q] = 0u;
        j[q] = 0u;
        if (b < L) {
            // first support index with s_j >= k0: from the bucket of k0, then
            // past the few supports between the bucket's start and k0
            const uint32_t *supp = st + (size_t)b * 2 * t;
            uint32_t lo = __ldg(first + (size_t)b * kLaneBuckets + (k0 >> lane_bshift(N)));
            uint32_t nx = lo < t ? __ldg(supp + lo) : 0xffffffffu;
            while (nx < k0) {
                ++lo;
                nx = lo < t ? __ldg(supp + lo) : 0xffffffffu;
            }
            j[q] = lo;
            next[q] = nx;
            cur[q] = __ldg(S + (size_t)b * (t + 1) + lo);
        }
    }
    for (uint32_t kb = k0; kb < k1; kb += 4) {  // k0 is a multiple of 4: 16-byte table loads
        uint32_t pk[4], vk[4];
        if (kb + 4 <= N) {
            const uint4 a = __ldg(reinterpret_cast<const uint4 *>(pi2 + kb));
            const uint4 c = __ldg(reinterpret_cast<const uint4 *>(v2m + kb));
            pk[0] = a.x; pk[1] = a.y; pk[2] = a.z; pk[3] = a.w;
            vk[0] = c.x; vk[1] = c.y; vk[2] = c.z; vk[3] = c.w;
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                pk[u] = kb + u < N ? __ldg(pi2 + kb + u) : 0u;
                vk[u] = kb + u < N ? __ldg(v2m + kb + u) : 0u;
            }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const uint32_t k = kb + u;
            if (k >= k1) break;
            uint32_t o[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint32_t b = 4 * g + q;
                while (next[q] < k) {
                    ++j[q];
                    next[q] = j[q] < t ? __ldg(st + (size_t)b * 2 * t + j[q]) : 0xffffffffu;
                    cur[q] = __ldg(S + (size_t)b * (t + 1) + j[q]);
                }
                o[q] = fmul_mont(cur[q], vk[u]);
            }
            C[(size_t)pk[u] * Lq + g] = make_uint4(o[0], o[1], o[2], o[3]);
        }
    }
}

// agg[tau][b] = sum over the tile's positions of C[i][b].
__global__ void __launch_bounds__(kLaneCta) k_lane_tile_sum(const uint4 *__restrict__ C, uint32_t N, uint32_t tile,
                                                           uint32_t L, uint4 *__restrict__ agg) {
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs come from the kernel before
    const uint32_t cols = lane_cols(L), Lq = lane_pad(L) / 4, ntiles = (N + tile - 1) / tile;
    const uint32_t g = blockIdx.y * cols + threadIdx.x % cols;
    const uint32_t tau = blockIdx.x * (kLaneCta / cols) + threadIdx.x / cols;
    if (g >= Lq || tau >= ntiles) return;
    const uint32_t i0 = tau * tile, i1 = min(N, i0 + tile);
    uint4 sum = make_uint4(0u, 0u, 0u, 0u);
    for (uint32_t i = i0; i < i1; i += 8) {
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
            v[u] = i + u < i1 ? C[(size_t)(i + u) * Lq + g] : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int u = 0; u < 8; ++u) sum = fadd4(sum, v[u]);
    }
    agg[(size_t)tau * Lq + g] = sum;
}

// carry[tau][b] = sum_{tau' > tau} agg[tau'][b]: one CTA per lane quad;
// thread c sums its chunk of consecutive tiles, a block-wide suffix scan of
// the chunk sums (warp shuffles, then the 32 warp totals) gives each chunk
// the sum of the tiles after it, and the thread writes its chunk's carries
// walking down.
__device__ __forceinline__ uint4 shfl_down4(uint4 v, int o) {
    return make_uint4(__shfl_down_sync(kFull, v.x, o), __shfl_down_sync(kFull, v.y, o),
                      __shfl_down_sync(kFull, v.z, o), __shfl_down_sync(kFull, v.w, o));
}
__device__ __forceinline__ uint4 fsub4(uint4 a, uint4 b) {
    return make_uint4(fsub(a.x, b.x), fsub(a.y, b.y), fsub(a.z, b.z), fsub(a.w, b.w));
}
__global__ void __launch_bounds__(kCarryThreads) k_lane_carry(const uint4 *__restrict__ agg, uint32_t ntiles,
                                                             uint32_t Lq, uint4 *__restrict__ carry) {
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs come from the kernel before
    __shared__ uint4 wsum[kCarryThreads / 32];
    const uint32_t g = blockIdx.x, c = threadIdx.x, lane = c & 31, warp = c >> 5;
    const uint32_t per = (ntiles + kCarryThreads - 1) / kCarryThreads;
    const uint32_t t0 = min(ntiles, c * per), t1 = min(ntiles, t0 + per);
    uint4 sum = make_uint4(0u, 0u, 0u, 0u);
    for (uint32_t tau = t0; tau < t1; tau += 8) {
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
            v[u] = tau + u < t1 ? agg[(size_t)(tau + u) * Lq + g] : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int u = 0; u < 8; ++u) sum = fadd4(sum, v[u]);
    }
    uint4 incl = sum;  // suffix within the warp: chunks lane .. 31
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint4 y = shfl_down4(incl, o);
        if (lane + o < 32) incl = fadd4(incl, y);
    }
    if (lane == 0) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {  // suffix over the warp totals
        const uint4 wv = wsum[lane];
        uint4 wi = wv;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint4 y = shfl_down4(wi, o);
            if (lane + o < 32) wi = fadd4(wi, y);
        }
        __syncwarp();
        wsum[lane] = fsub4(wi, wv);  // totals of the warps after this one
    }
    __syncthreads();
    uint4 run = fadd4(fsub4(incl, sum), wsum[warp]);  // sum over the chunks after this one
    for (uint32_t hi = t1; hi > t0;) {  // eight tiles at a time, loads first
        const uint32_t cnt = hi - t0 < 8u ? hi - t0 : 8u;
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
            v[u] = (uint32_t)u < cnt ? agg[(size_t)(hi - 1 - u) * Lq + g] : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            if ((uint32_t)u < cnt) {
                carry[(size_t)(hi - 1 - u) * Lq + g] = run;
                run = fadd4(run, v[u]);
            }
        }
        hi -= cnt;
    }
}

// In place: C[i][b] <- v1_i (carry[tau][b] + sum_{i' >= i in tile tau} C[i'][b]),
// with v1m = v1 R (Montgomery, R = 2^32) so that each product is one REDC.
__global__ void __launch_bounds__(kLaneCta, 4) k_lane_scan(uint4 *__restrict__ C, uint32_t N, uint32_t tile, uint32_t L,
                                                       const uint4 *__restrict__ carry,
                                                       const uint32_t *__restrict__ v1m) {
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs come from the kernel before
    const uint32_t cols = lane_cols(L), Lq = lane_pad(L) / 4, ntiles = (N + tile - 1) / tile;
    const uint32_t g = blockIdx.y * cols + threadIdx.x % cols;
    const uint32_t tau = blockIdx.x * (kLaneCta / cols) + threadIdx.x / cols;
    if (g >= Lq || tau >= ntiles) return;
    const uint32_t i0 = tau * tile, i1 = min(N, i0 + tile);
    uint4 run = carry[(size_t)tau * Lq + g];
    for (uint32_t hi = i1; hi > i0;) {
        const uint32_t cnt = hi - i0 < 8u ? hi - i0 : 8u;  // positions hi-1 .. hi-cnt
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
            v[u] = (uint32_t)u < cnt ? C[(size_t)(hi - 1 - u) * Lq + g] : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            if ((uint32_t)u < cnt) {
                const uint32_t i = hi - 1 - u, w = __ldg(v1m + i);
                run = fadd4(run, v[u]);
                C[(size_t)i * Lq + g] = make_uint4(fmul_mont(run.x, w), fmul_mont(run.y, w), fmul_mont(run.z, w),
                                                   fmul_mont(run.w, w));
            }
        }
        hi -= cnt;
    }
}

// out[b][j] = addend[b][j] + sum_{c<r} C[pi1^-1(r j + c)][b] for kGatherJ
// outputs and the CTA's lanes, transposed through shared memory so that out
// rows are written 128 bytes at a time.  addend may be null or alias out.
__global__ void __launch_bounds__(kLaneCta, 4) k_lane_gather(const uint4 *__restrict__ C,
                                                         const uint32_t *__restrict__ pi1inv,
                                                         uint32_t r, uint32_t n, uint32_t L,
                                                         const uint32_t *addend, uint32_t *out) {
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs come from the kernel before
    __shared__ uint32_t tile[kGatherJ][4 * kLaneQuadsMax + 1];
    const uint32_t cols = lane_cols(L), subs = kLaneCta / cols, Lq = lane_pad(L) / 4;
    const uint32_t tid = threadIdx.x, gl = tid % cols, sub = tid / cols;
    const uint32_t g = blockIdx.y * cols + gl;
    const uint32_t j0 = blockIdx.x * kGatherJ;
    // thread (sub, quad) takes outputs jj = sub, sub + subs, ... two at a time
    for (uint32_t jj0 = sub; jj0 < (uint32_t)kGatherJ; jj0 += 2 * subs) {
        uint4 v[2][8];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const uint32_t jj = jj0 + q * subs, j = j0 + jj;
            const bool ok = jj < (uint32_t)kGatherJ && j < n && g < Lq;
#pragma unroll
            for (int c = 0; c < 8; ++c)
                v[q][c] = ok && (uint32_t)c < r ? C[(size_t)__ldg(pi1inv + (size_t)j * r + c) * Lq + g]
                                              : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const uint32_t jj = jj0 + q * subs, j = j0 + jj;
            if (jj >= (uint32_t)kGatherJ) continue;
            uint4 acc = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int c = 0; c < 8; ++c) acc = fadd4(acc, v[q][c]);
            if (r > 8 && j < n && g < Lq)
                for (uint32_t c = 8; c < r; ++c)
                    acc = fadd4(acc, C[(size_t)__ldg(pi1inv + (size_t)j * r + c) * Lq + g]);
            tile[jj][4 * gl] = acc.x;
            tile[jj][4 * gl + 1] = acc.y;
            tile[jj][4 * gl + 2] = acc.z;
            tile[jj][4 * gl + 3] = acc.w;
        }
    }
    __syncthreads();
    // consecutive threads write consecutive outputs of one vector's row
    for (uint32_t idx = tid; idx < 4 * cols * (uint32_t)kGatherJ; idx += kLaneCta) {
        const uint32_t bb = idx / kGatherJ, jj = idx % kGatherJ;
        const uint32_t vb = blockIdx.y * 4 * cols + bb, j = j0 + jj;
        if (vb < L && j < n) {
            const size_t o = (size_t)vb * n + j;
            out[o] = addend ? fadd(addend[o], tile[jj][bb]) : tile[jj][bb];
        }
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
    const cudaError_t attr = func_attr((const void *)k_sample_sparse, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kSampleMaxSmem);
    if (attr != cudaSuccess) return attr;
    k_sample_sparse<<<count, 32, smem, s>>>(key, tag, idx0, N, t, out, clear, clear_words); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_syndrome_scan(const uint32_t *pi2inv, const uint32_t *v2p, const uint32_t *v1,
                                 uint32_t N, const uint32_t *sparse, uint32_t t, uint32_t count,
                                 uint32_t *F, unsigned long long *status, uint32_t *err,
                                 cudaStream_t s) {
    if (count == 0) return cudaSuccess;
    const size_t smem = (2 * (size_t)t + 1) * sizeof(uint32_t);
    const unsigned grid = count * scan_tiles(N);
    const DebugWait dbg = debug_wait();
    const bool inject = dbg.site == PVMVMD_DEBUG_WAIT_SCAN;
    k_syndrome_scan<<<grid, kScanThreads, smem, s>>>(pi2inv, v2p, v1, N, sparse, t, count, F, status,
                                                     err, inject ? dbg.index : 0xFFFFFFFFu,
                                                     inject ? (uint32_t)dbg.limit : kSpinLimit); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_syndrome_gather(const uint32_t *pi1inv, uint32_t n, uint32_t r,
                                   const uint32_t *F, uint32_t N, const uint32_t *addend,
                                   uint32_t *out, uint32_t count, cudaStream_t s) {
    if (count == 0 || n == 0) return cudaSuccess;
    dim3 grid((n + 255) / 256, count);
    k_syndrome_gather<<<grid, 256, 0, s>>>(pi1inv, n, r, F, N, addend, out); note_launch();
    return cudaGetLastError();
}

size_t encode_scan_status_words(uint32_t N, uint32_t L) {
    return (size_t)((L + 255) / 256) * ((N + kEncTile - 1) / kEncTile) * 256;
}

cudaError_t encode_scan_clear(unsigned long long *status, uint32_t *ticket, uint32_t N, uint32_t L,
                              cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(status, 0, encode_scan_status_words(N, L) * sizeof(unsigned long long), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(ticket, 0, sizeof(uint32_t), s);
    return e;
}

cudaError_t launch_encode_scan(const void *X, bool x_is_i8, size_t ldx, const uint32_t *perm,
                               uint32_t div, const uint32_t *vscale_m, uint32_t N, uint32_t L,
                               uint32_t *Y, size_t ldy, unsigned long long *status, uint32_t *ticket,
                               uint32_t *err, cudaStream_t s) {
    const size_t ctas = encode_scan_status_words(N, L) / 256;
    if (ctas == 0) return cudaSuccess;
    if (ctas > 0x7fffffffu) return cudaErrorInvalidValue;
    if (x_is_i8)
        k_encode_scan<true><<<(unsigned)ctas, 256, 0, s>>>(X, ldx, perm, div, vscale_m, N, L, Y, ldy,
                                                           status, ticket, err);
    else
        k_encode_scan<false><<<(unsigned)ctas, 256, 0, s>>>(X, ldx, perm, div, vscale_m, N, L, Y, ldy,
                                                            status, ticket, err);
    note_launch();
    return cudaGetLastError();
}

cudaError_t launch_transpose_i8(const int8_t *in, int R, int C, int8_t *out, cudaStream_t s) {
    if (R <= 0 || C <= 0) return cudaSuccess;
    dim3 grid((C + 31) / 32, (R + 31) / 32), block(32, 8);
    if (grid.y > 65535u) return cudaErrorInvalidValue;
    k_transpose_i8<<<grid, block, 0, s>>>(in, R, C, out); note_launch();
    return cudaGetLastError();
}


namespace {
uint32_t fused_slice(uint32_t N, int C) {
    return (uint32_t)(((N + C - 1) / C + kFusedThreads - 1) / kFusedThreads) * kFusedThreads;
}
size_t fused_smem(uint32_t slice, uint32_t t) {
    return ((size_t)slice + slice / 32 + 3 * (size_t)t + 1 + 1024) * sizeof(uint32_t);
}
constexpr size_t kFusedMaxSmem = 180 * 1024;

}  // namespace

// Cluster size and slice for the fused syndrome; false if N is too long for
// one cluster of at most 8 CTAs.
bool syndrome_fused_plan(uint32_t N, uint32_t t, int *C_out, uint32_t *slice_out, size_t *smem_out) {
    // one CTA when the padded intermediate fits, else the smallest cluster
    for (int C = 1; C <= 8; C *= 2) {
        const uint32_t slice = fused_slice(N, C);
        const size_t smem = fused_smem(slice, t);
        if (smem <= kFusedMaxSmem) {
            *C_out = C;
            *slice_out = slice;
            *smem_out = smem;
            return true;
        }
    }
    return false;
}

// The cluster size one launch of `count` vectors uses: the smallest that
// holds the intermediate, and for a batch that leaves most SMs idle (at most
// a quarter busy) doubled while count * C * spread CTAs still fit the SMs
// and every CTA keeps at least one position per thread, up to 8 CTAs.  A
// small batch then spreads each vector's serial work over a few SMs instead
// of one; larger batches keep the cheaper per-position work of the smallest
// cluster.  The callers' spread (launch_syndrome_fused) was measured: 4 for
// encodes (8 vectors per call: Qwen3-4B block 0.265 -> 0.227 ms per step
// against spread 1; 2 gave 0.275, 8 gave 0.255); for the ell = 2 shared
// challenges 16 when the batch is large (a cluster of at most 2 CTAs at
// N_y = 32768, taking few SMs from the decrypt beside it: batch-1 workload of
// 100 vectors 0.3256 -> 0.3220 ms per step against spread 4), else 4 (the
// challenges are then the decode's critical path: Qwen3-4B block, 8
// vectors, 0.227 against 0.235 ms; one token with its 448 single-vector
// encodes and decodes, client part 9.7 against 10.2 ms).  (Up to 16 CTAs, a
// non-portable size, made one decode call alone slightly faster, 0.3228
// against 0.3242 ms per batch-1 step, but a layer's decodes side by side
// fit only seven 16-CTA clusters at once: 8B layer, 64 vectors, 0.528
// against 0.506 ms per step; Qwen3-4B block, 8 vectors, 0.324 against
// 0.266 ms.)
constexpr int kFusedClusterMax = 8;
static void syndrome_fused_launch_plan(uint32_t N, uint32_t t, uint32_t count, int *C, uint32_t *slice,
                                       size_t *smem, int spread) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if ((uint64_t)count * (uint64_t)*C * 4 > (uint64_t)sms) return;
    const int cmax = kFusedClusterMax;
    while (*C < cmax && (uint64_t)count * (uint64_t)(2 * *C) * (uint64_t)spread <= (uint64_t)sms &&
           (uint64_t)(2 * *C) * kFusedThreads <= (uint64_t)N) {
        *C *= 2;
        *slice = fused_slice(N, *C);
        *smem = fused_smem(*slice, t);
    }
}

cudaError_t launch_syndrome_fused(const pvmvmd_key &key, uint32_t tag, uint64_t idx0, uint32_t N,
                                  uint32_t t, uint32_t count, const uint32_t *pi2inv,
                                  const uint32_t *v2p, const uint32_t *v1, const uint32_t *pi1inv,
                                  const uint32_t *pi2, const uint32_t *v2m, const uint32_t *v1pm,
                                  uint32_t n, uint32_t r, uint32_t *sparse_out,
                                  const uint32_t *addend, uint32_t *out, cudaStream_t s, bool pdl,
                                  int spread) {
    if (count == 0) return cudaSuccess;
    int C = 0;
    uint32_t slice = 0;
    size_t smem = 0;
    if (!syndrome_fused_plan(N, t, &C, &slice, &smem)) return cudaErrorNotSupported;
    const cudaError_t attr = func_attr((const void *)k_syndrome_fused, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kFusedMaxSmem);
    if (attr != cudaSuccess) return attr;
    syndrome_fused_launch_plan(N, t, count < 65535 ? count : 65535, &C, &slice, &smem, spread < 1 ? 1 : spread);
    for (uint32_t c0 = 0; c0 < count; c0 += 65535) {
        const uint32_t nb = count - c0 < 65535 ? count - c0 : 65535;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(C, nb, 1);
        cfg.blockDim = dim3(kFusedThreads, 1, 1);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = s;
        cudaLaunchAttribute attr1[2];
        attr1[0].id = cudaLaunchAttributeClusterDimension;
        attr1[0].val.clusterDim.x = C;
        attr1[0].val.clusterDim.y = 1;
        attr1[0].val.clusterDim.z = 1;
        attr1[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr1[1].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr1;
        cfg.numAttrs = pdl ? 2 : 1;
        cudaError_t e = counted_launch(cudaLaunchKernelEx(&cfg, k_syndrome_fused, key, tag, idx0 + c0, N, t, slice,
                                           pi2inv, v2p, v1, pi1inv, n, r,
                                           sparse_out + (size_t)c0 * 2 * t,
                                           addend ? addend + (size_t)c0 * n : nullptr,
                                           out + (size_t)c0 * n, pi2, v2m, v1pm));
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

namespace {
cudaError_t launch_pdl(const void *fn, dim3 grid, dim3 block, size_t smem, cudaStream_t s, void **args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute a[1];
    a[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    a[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = a;
    cfg.numAttrs = 1;
    return counted_launch(cudaLaunchKernelExC(&cfg, fn, args));
}
}  // namespace

size_t lane_state_words(uint32_t t, uint32_t L) {
    return (size_t)L * (t + 1) + (size_t)L * kLaneBuckets / 2;
}

size_t lane_aux_words(uint32_t N, uint32_t L) {
    return 2 * (size_t)((N + kLaneTileMin - 1) / kLaneTileMin) * lane_pad(L);
}

cudaError_t launch_lane_syndrome(const pvmvmd_key &key, uint32_t tag, uint64_t idx0, uint32_t N,
                                 uint32_t t, uint32_t L, const uint32_t *pi2, const uint32_t *v2m,
                                 const uint32_t *v1m, const uint32_t *pi1inv, uint32_t n, uint32_t r,
                                 uint32_t *sparse_out, uint32_t *S, uint32_t *C, uint32_t *aux,
                                 const uint32_t *addend, uint32_t *out, cudaStream_t s) {
    if (L == 0) return cudaSuccess;
    const size_t smem = ((size_t)(N + 31) / 32 + 1024 + 4 * (size_t)t + 1) * sizeof(uint32_t);
    if (smem > kSampleMaxSmem) return cudaErrorInvalidValue;
    const cudaError_t a1 = func_attr((const void *)k_lane_sample, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)kSampleMaxSmem);
    if (a1 != cudaSuccess) return a1;
    if ((reinterpret_cast<uintptr_t>(C) | reinterpret_cast<uintptr_t>(aux)) & 15u)
        return cudaErrorInvalidValue;
    const uint32_t Lp = lane_pad(L), cols = lane_cols(L), per_cta = kLaneCta / cols;
    const unsigned gy = (Lp / 4 + cols - 1) / cols;
    // tiles of 32 positions, or 64 / 128 when the tile-sum and scan grids
    // still hold two CTAs of threads per SM: longer tiles shorten the carry
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    uint32_t tile = kLaneTileMin;
    while (tile < (uint32_t)kLaneTileMax &&
           (uint64_t)((N + 2 * tile - 1) / (2 * tile)) * (lane_pad(L) / 4) >= (uint64_t)2 * sms * kLaneCta)
        tile *= 2;
    const uint32_t ntiles = (N + tile - 1) / tile;
    const uint32_t nspans = (N + kExpandSpan - 1) / kExpandSpan;
    if (gy > 65535u || L > 0x7fffffffu) return cudaErrorInvalidValue;
    uint4 *agg = reinterpret_cast<uint4 *>(aux), *carry = reinterpret_cast<uint4 *>(aux + (size_t)ntiles * Lp);
    uint4 *C4 = reinterpret_cast<uint4 *>(C);
    const uint4 *C4c = C4, *aggc = agg, *carryc = carry;
    const uint32_t Lq = Lp / 4;
    const uint32_t *stc = sparse_out, *Sc = S;
    // S holds the suffix sums [L][t+1], then the bucket index [L][kLaneBuckets] (uint16)
    uint16_t *first = reinterpret_cast<uint16_t *>(S + (size_t)L * (t + 1));
    const uint16_t *fc = first;
    cudaError_t e;
    void *a0[] = {(void *)&key, &tag, &idx0, &N, &t, &sparse_out, &S, &first};
    if ((e = launch_pdl((const void *)k_lane_sample, dim3(L), dim3(128), smem, s, a0)) != cudaSuccess) return e;
    void *a1x[] = {&stc, &Sc, &fc, &t, &N, &L, (void *)&pi2, (void *)&v2m, &C4};
    if ((e = launch_pdl((const void *)k_lane_expand, dim3((nspans + per_cta - 1) / per_cta, gy), dim3(kLaneCta), 0, s,
                        a1x)) != cudaSuccess)
        return e;
    void *a2[] = {&C4c, &N, &tile, &L, &agg};
    if ((e = launch_pdl((const void *)k_lane_tile_sum, dim3((ntiles + per_cta - 1) / per_cta, gy), dim3(kLaneCta), 0,
                        s, a2)) != cudaSuccess)
        return e;
    void *a3[] = {&aggc, (void *)&ntiles, (void *)&Lq, &carry};
    if ((e = launch_pdl((const void *)k_lane_carry, dim3(Lq), dim3(kCarryThreads), 0, s, a3)) != cudaSuccess) return e;
    void *a4[] = {&C4, &N, &tile, &L, &carryc, (void *)&v1m};
    if ((e = launch_pdl((const void *)k_lane_scan, dim3((ntiles + per_cta - 1) / per_cta, gy), dim3(kLaneCta), 0, s,
                        a4)) != cudaSuccess)
        return e;
    void *a5[] = {&C4c, (void *)&pi1inv, &r, &n, &L, (void *)&addend, &out};
    if ((e = launch_pdl((const void *)k_lane_gather, dim3((n + kGatherJ - 1) / kGatherJ, gy), dim3(kLaneCta), 0, s,
                        a5)) != cudaSuccess)
        return e;
    return cudaGetLastError();
}

}  // namespace pv
