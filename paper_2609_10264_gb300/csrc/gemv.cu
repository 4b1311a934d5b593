// Batch-1 field GEMV: y_hat = M x_hat over F_q (the server's online work,
// Sec. 6.1), M int8 m x K row-major, x_hat canonical uint32.
//
// Design (bandwidth-bound; one byte of M per field MAC):
//  * Each CTA splits x_hat once into four signed base-256 digit planes in
//    shared memory (x_hat centred = d0 + 2^8 d1 + 2^16 d2 + 2^24 d3), so a
//    field MAC becomes four int8 x int8 products done by dp4a, four columns
//    per instruction, with exact int32 sums (|sum| <= 128*128*K < 2^31).
//  * M streams through 128-bit non-allocating loads; a warp owns ROWS rows at
//    a time and walks their columns 512 at a time (16 bytes per lane), with
//    the next batch's loads issued before the current batch's arithmetic.
//  * Row groups are dealt round-robin over CTAs first, so every SM gets an
//    equal share of rows whatever m is.
//  * Per row: a transposed butterfly reduces the 4*ROWS lane partials in
//    4*ROWS - 1 + log2(32/(4*ROWS)) shuffles, the four limb sums are combined
//    in int64 and reduced mod q once.
#include <algorithm>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "launch.h"

namespace pv {
namespace {

constexpr int kGemvThreads = 512;
// Digit planes of a K segment live in shared memory (4 bytes per column); a
// longer K is done in segments whose mod-q partial results are added.
constexpr int kGemvMaxK = 48 * 1024;

__device__ __forceinline__ uint4 ldg_stream(const void *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// 16 bytes of row `row` starting at column 16*chunk, zero-filled past K.
template <bool kVec>
__device__ __forceinline__ uint4 load_chunk(const int8_t *__restrict__ W, size_t ldw, size_t row,
                                            int K, int chunk) {
    const int8_t *p = W + row * ldw + (size_t)chunk * 16;
    if (kVec) return ldg_stream(p);
    uint32_t w[4] = {0u, 0u, 0u, 0u};
    const int c0 = chunk * 16;
#pragma unroll
    for (int b = 0; b < 16; ++b)
        if (c0 + b < K) w[b >> 2] |= (uint32_t)(uint8_t)__ldg(p + b) << (8 * (b & 3));
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// Sum of v[index] over the 32 lanes, where index = lane / (32 / V): after the
// call every lane holds the total of the entry its lane number selects.
template <int V>
__device__ __forceinline__ int transposed_reduce(int (&v)[V], int lane) {
#pragma unroll
    for (int n = V, o = 16; n > 1; n >>= 1, o >>= 1) {
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < n / 2; ++i) {
            const int send = upper ? v[i] : v[i + n / 2];
            const int keep = upper ? v[i + n / 2] : v[i];
            v[i] = keep + __shfl_xor_sync(kFull, send, o);
        }
    }
    int x = v[0];
#pragma unroll
    for (int o = 16 / V; o >= 1; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
    return x;
}

template <int ROWS, int UNROLL, bool kVec>
__global__ void __launch_bounds__(kGemvThreads, 1)
    k_gemv(const int8_t *__restrict__ W, size_t ldw, int m, int K, const uint32_t *__restrict__ xhat,
           uint32_t *__restrict__ y, bool accumulate) {
    extern __shared__ uint4 s_planes[];  // 4 planes of nchunks 16-byte chunks
    const int nchunks = (K + 15) / 16;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr int nwarps = kGemvThreads / 32;
    constexpr int V = ROWS * 4;
    static_assert(V <= 32 && (V & (V - 1)) == 0, "ROWS must be 1, 2, 4 or 8");

    const int ngroups = (m + ROWS - 1) / ROWS;
    const int gstride = gridDim.x * nwarps;
    int g = warp * gridDim.x + blockIdx.x;

    // Issue the first batch of M loads before building the digit planes.
    uint4 wbuf[UNROLL][ROWS];
    auto issue = [&](int grp, int c) {
#pragma unroll
        for (int u = 0; u < UNROLL; ++u)
#pragma unroll
            for (int r = 0; r < ROWS; ++r) {
                const int cc = c + 32 * u, row = grp * ROWS + r;
                wbuf[u][r] = (cc < nchunks && row < m) ? load_chunk<kVec>(W, ldw, (size_t)row, K, cc)
                                                       : make_uint4(0u, 0u, 0u, 0u);
            }
    };
    if (g < ngroups) issue(g, lane);

    // Digit planes of x_hat (zero past K).
    uint32_t *planes = reinterpret_cast<uint32_t *>(s_planes);
    const int pstride = nchunks * 4;  // words per plane
    for (int q4 = tid; q4 < pstride; q4 += kGemvThreads) {
        uint32_t p0 = 0, p1 = 0, p2 = 0, p3 = 0;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int k = q4 * 4 + b;
            if (k < K) {
                int d0, d1, d2, d3;
                limb_split(__ldg(xhat + k), d0, d1, d2, d3);
                p0 |= (uint32_t)(d0 & 0xff) << (8 * b);
                p1 |= (uint32_t)(d1 & 0xff) << (8 * b);
                p2 |= (uint32_t)(d2 & 0xff) << (8 * b);
                p3 |= (uint32_t)(d3 & 0xff) << (8 * b);
            }
        }
        planes[q4] = p0;
        planes[pstride + q4] = p1;
        planes[2 * pstride + q4] = p2;
        planes[3 * pstride + q4] = p3;
    }
    __syncthreads();
    const uint4 *P0 = s_planes, *P1 = s_planes + nchunks, *P2 = s_planes + 2 * nchunks,
                *P3 = s_planes + 3 * nchunks;

    for (; g < ngroups; g += gstride) {
        int acc[ROWS][4];
#pragma unroll
        for (int r = 0; r < ROWS; ++r) acc[r][0] = acc[r][1] = acc[r][2] = acc[r][3] = 0;

        for (int c = lane; c < nchunks; c += 32 * UNROLL) {
            uint4 cur[UNROLL][ROWS];
#pragma unroll
            for (int u = 0; u < UNROLL; ++u)
#pragma unroll
                for (int r = 0; r < ROWS; ++r) cur[u][r] = wbuf[u][r];
            // prefetch: the next column batch of this group, else the next group
            const int cn = c + 32 * UNROLL;
            if (cn < nchunks) issue(g, cn);
            else if (g + gstride < ngroups) issue(g + gstride, lane);
#pragma unroll
            for (int u = 0; u < UNROLL; ++u) {
                const int cc = c + 32 * u;
                if (cc < nchunks) {
                    const uint4 l0 = P0[cc], l1 = P1[cc], l2 = P2[cc], l3 = P3[cc];
#pragma unroll
                    for (int r = 0; r < ROWS; ++r) {
                        const uint4 w = cur[u][r];
                        acc[r][0] = __dp4a((int)w.x, (int)l0.x, acc[r][0]);
                        acc[r][1] = __dp4a((int)w.x, (int)l1.x, acc[r][1]);
                        acc[r][2] = __dp4a((int)w.x, (int)l2.x, acc[r][2]);
                        acc[r][3] = __dp4a((int)w.x, (int)l3.x, acc[r][3]);
                        acc[r][0] = __dp4a((int)w.y, (int)l0.y, acc[r][0]);
                        acc[r][1] = __dp4a((int)w.y, (int)l1.y, acc[r][1]);
                        acc[r][2] = __dp4a((int)w.y, (int)l2.y, acc[r][2]);
                        acc[r][3] = __dp4a((int)w.y, (int)l3.y, acc[r][3]);
                        acc[r][0] = __dp4a((int)w.z, (int)l0.z, acc[r][0]);
                        acc[r][1] = __dp4a((int)w.z, (int)l1.z, acc[r][1]);
                        acc[r][2] = __dp4a((int)w.z, (int)l2.z, acc[r][2]);
                        acc[r][3] = __dp4a((int)w.z, (int)l3.z, acc[r][3]);
                        acc[r][0] = __dp4a((int)w.w, (int)l0.w, acc[r][0]);
                        acc[r][1] = __dp4a((int)w.w, (int)l1.w, acc[r][1]);
                        acc[r][2] = __dp4a((int)w.w, (int)l2.w, acc[r][2]);
                        acc[r][3] = __dp4a((int)w.w, (int)l3.w, acc[r][3]);
                    }
                }
            }
        }

        int v[V];
#pragma unroll
        for (int r = 0; r < ROWS; ++r)
#pragma unroll
            for (int p = 0; p < 4; ++p) v[r * 4 + p] = acc[r][p];
        const int tot = transposed_reduce<V>(v, lane);
        // lane l holds entry l / (32/V) = 4 r + p
        constexpr int span = 32 / V;
        const int a1 = __shfl_down_sync(kFull, tot, span);
        const int a2 = __shfl_down_sync(kFull, tot, 2 * span);
        const int a3 = __shfl_down_sync(kFull, tot, 3 * span);
        const int entry = lane / span;
        if ((lane % span) == 0 && (entry & 3) == 0) {
            const int row = g * ROWS + (entry >> 2);
            if (row < m) {
                const int64_t s = (int64_t)tot + ((int64_t)a1 << 8) + ((int64_t)a2 << 16) +
                                  ((int64_t)a3 << 24);
                const uint32_t part = fred_signed(s);
                y[row] = accumulate ? fadd(y[row], part) : part;
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Grouped persistent variant (K % 16 == 0, 16-byte aligned rows): one launch
// computes a list of independent batch-1 products (jobs), each streaming its
// own matrix once.  The bytes of all matrices are split evenly over the CTAs
// (whole rows); a CTA walks its share job by job, splitting that job's x_hat
// into digit planes once, and its warps stream row pairs with the loads of
// the next batch issued before the arithmetic of the current one (and, on
// long streams, a bulk L2 prefetch of its next row group).  A single
// launch over many matrices keeps every SM's loads in flight for the whole
// stream instead of paying the ramp-up and drain of one launch per matrix.
// Launched with programmatic dependent launch; it waits for the preceding
// kernel (griddepcontrol.wait) before reading anything.
// ---------------------------------------------------------------------------
constexpr int kMultiThreads = 256;
constexpr int kMultiWarps = kMultiThreads / 32;

struct MultiArgs {
    int count;
    long long base[kMultiMaxJobs + 1];  // prefix sums of m_j * K_j (bytes of M)
    MvmJob job[kMultiMaxJobs];
};

// kPrefetch: warps ask L2 for their next group of rows (long streams only).
template <int ROWS, int UNROLL, bool kPrefetch>
__global__ void __launch_bounds__(kMultiThreads, 2) k_gemv_multi(const __grid_constant__ MultiArgs args) {
    extern __shared__ uint4 s_planes[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr int V = ROWS * 4;
    const long long total = args.base[args.count];
    const long long lo = total * blockIdx.x / gridDim.x;
    const long long hi = total * (blockIdx.x + 1) / gridDim.x;

    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    // The first loads of M go out before griddepcontrol.wait, so they overlap
    // the end of the kernel before this one: M is the server's weight
    // matrix, never written by a kernel that signals its dependents early.
    // Everything else (x_hat, y_hat) is touched only after the wait.
    bool waited = false;

    for (int j = 0; j < args.count; ++j) {
        const long long b0 = args.base[j], b1 = args.base[j + 1];
        if (b1 <= lo || b0 >= hi) continue;
        const MvmJob &job = args.job[j];
        const int K = job.K, m = job.m, nchunks = K / 16;
        // rows whose first byte lies in [lo, hi)
        const int row_a = lo > b0 ? (int)((lo - b0 + K - 1) / K) : 0;
        const int row_b = (int)min((long long)m, (hi - b0 + K - 1) / K);
        if (row_a >= row_b) continue;
        const int ngroups = (row_b - row_a + ROWS - 1) / ROWS;

        uint4 wbuf[UNROLL][ROWS];
        auto issue = [&](int grp, int c) {
#pragma unroll
            for (int u = 0; u < UNROLL; ++u)
#pragma unroll
                for (int r = 0; r < ROWS; ++r) {
                    const int cc = c + 32 * u, row = row_a + grp * ROWS + r;
                    wbuf[u][r] = (cc < nchunks && row < row_b)
                                     ? ldg_stream(job.W + (size_t)row * job.ldw + (size_t)cc * 16)
                                     : make_uint4(0u, 0u, 0u, 0u);
                }
        };
        int g = warp;
        if (g < ngroups) issue(g, lane);
        if (!waited) {
            asm volatile("griddepcontrol.wait;" ::: "memory");
            waited = true;
        }

        __syncthreads();  // the previous job's planes are no longer read
        uint32_t *planes = reinterpret_cast<uint32_t *>(s_planes);
        const int pstride = K / 4;
        for (int q4 = tid; q4 < pstride; q4 += kMultiThreads) {
            const uint4 xv = __ldg(reinterpret_cast<const uint4 *>(job.xhat) + q4);
            const uint32_t xs[4] = {xv.x, xv.y, xv.z, xv.w};
            uint32_t p0 = 0, p1 = 0, p2 = 0, p3 = 0;
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                int d0, d1, d2, d3;
                limb_split(xs[b], d0, d1, d2, d3);
                p0 |= (uint32_t)(d0 & 0xff) << (8 * b);
                p1 |= (uint32_t)(d1 & 0xff) << (8 * b);
                p2 |= (uint32_t)(d2 & 0xff) << (8 * b);
                p3 |= (uint32_t)(d3 & 0xff) << (8 * b);
            }
            planes[q4] = p0;
            planes[pstride + q4] = p1;
            planes[2 * pstride + q4] = p2;
            planes[3 * pstride + q4] = p3;
        }
        __syncthreads();
        const uint4 *P0 = s_planes, *P1 = s_planes + nchunks, *P2 = s_planes + 2 * nchunks,
                    *P3 = s_planes + 3 * nchunks;

        for (; g < ngroups; g += kMultiWarps) {
            if (kPrefetch && lane < ROWS && g + kMultiWarps < ngroups) {
                // the rows of this warp's next group, whole, into L2 while
                // this group streams through the registers
                const int row = row_a + (g + kMultiWarps) * ROWS + lane;
                if (row < row_b)
                    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(job.W + (size_t)row * job.ldw),
                                 "r"((uint32_t)K)
                                 : "memory");
            }
            int acc[ROWS][4];
#pragma unroll
            for (int r = 0; r < ROWS; ++r) acc[r][0] = acc[r][1] = acc[r][2] = acc[r][3] = 0;
            for (int c = lane; c < nchunks; c += 32 * UNROLL) {
                uint4 cur[UNROLL][ROWS];
#pragma unroll
                for (int u = 0; u < UNROLL; ++u)
#pragma unroll
                    for (int r = 0; r < ROWS; ++r) cur[u][r] = wbuf[u][r];
                const int cn = c + 32 * UNROLL;
                if (cn < nchunks) issue(g, cn);
                else if (g + kMultiWarps < ngroups) issue(g + kMultiWarps, lane);
#pragma unroll
                for (int u = 0; u < UNROLL; ++u) {
                    const int cc = c + 32 * u;
                    if (cc < nchunks) {
                        const uint4 l0 = P0[cc], l1 = P1[cc], l2 = P2[cc], l3 = P3[cc];
#pragma unroll
                        for (int r = 0; r < ROWS; ++r) {
                            const uint4 w = cur[u][r];
                            acc[r][0] = __dp4a((int)w.x, (int)l0.x, acc[r][0]);
                            acc[r][1] = __dp4a((int)w.x, (int)l1.x, acc[r][1]);
                            acc[r][2] = __dp4a((int)w.x, (int)l2.x, acc[r][2]);
                            acc[r][3] = __dp4a((int)w.x, (int)l3.x, acc[r][3]);
                            acc[r][0] = __dp4a((int)w.y, (int)l0.y, acc[r][0]);
                            acc[r][1] = __dp4a((int)w.y, (int)l1.y, acc[r][1]);
                            acc[r][2] = __dp4a((int)w.y, (int)l2.y, acc[r][2]);
                            acc[r][3] = __dp4a((int)w.y, (int)l3.y, acc[r][3]);
                            acc[r][0] = __dp4a((int)w.z, (int)l0.z, acc[r][0]);
                            acc[r][1] = __dp4a((int)w.z, (int)l1.z, acc[r][1]);
                            acc[r][2] = __dp4a((int)w.z, (int)l2.z, acc[r][2]);
                            acc[r][3] = __dp4a((int)w.z, (int)l3.z, acc[r][3]);
                            acc[r][0] = __dp4a((int)w.w, (int)l0.w, acc[r][0]);
                            acc[r][1] = __dp4a((int)w.w, (int)l1.w, acc[r][1]);
                            acc[r][2] = __dp4a((int)w.w, (int)l2.w, acc[r][2]);
                            acc[r][3] = __dp4a((int)w.w, (int)l3.w, acc[r][3]);
                        }
                    }
                }
            }
            int v[V];
#pragma unroll
            for (int r = 0; r < ROWS; ++r)
#pragma unroll
                for (int p = 0; p < 4; ++p) v[r * 4 + p] = acc[r][p];
            const int tot = transposed_reduce<V>(v, lane);
            constexpr int span = 32 / V;
            const int a1 = __shfl_down_sync(kFull, tot, span);
            const int a2 = __shfl_down_sync(kFull, tot, 2 * span);
            const int a3 = __shfl_down_sync(kFull, tot, 3 * span);
            const int entry = lane / span;
            if ((lane % span) == 0 && (entry & 3) == 0) {
                const int row = row_a + g * ROWS + (entry >> 2);
                if (row < row_b) {
                    const int64_t sum = (int64_t)tot + ((int64_t)a1 << 8) + ((int64_t)a2 << 16) +
                                        ((int64_t)a3 << 24);
                    const uint32_t part = fred_signed(sum);
                    job.y[row] = job.accumulate ? fadd(job.y[row], part) : part;
                }
            }
        }
    }
    if (!waited) asm volatile("griddepcontrol.wait;" ::: "memory");
}

cudaError_t run_gemv_multi(const MvmJob *jobs, int count, cudaStream_t s) {
    static MultiArgs args;  // host staging of the kernel parameters (copied at launch)
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    args.count = count;
    args.base[0] = 0;
    int kmax = 16;
    for (int j = 0; j < count; ++j) {
        args.job[j] = jobs[j];
        args.base[j + 1] = args.base[j] + (long long)jobs[j].m * jobs[j].K;
        if (jobs[j].K > kmax) kmax = jobs[j].K;
    }
    long long rows = 0;
    for (int j = 0; j < count; ++j) rows += jobs[j].m;
    if (rows == 0) return cudaSuccess;
    for (const void *f : {(const void *)k_gemv_multi<2, 4, false>, (const void *)k_gemv_multi<2, 4, true>}) {
        const cudaError_t attr = func_attr(f, cudaFuncAttributeMaxDynamicSharedMemorySize, 4 * kMultiMaxK);
        if (attr != cudaSuccess) return attr;
    }
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    long long grid = 2LL * sms;
    if (grid > rows) grid = rows;
    // The L2 prefetch of each warp's next row group pays on long streams
    // (100 requests of 4096 x 4096 per launch: GEMV 269.7 -> 261.2 us) and
    // costs on short ones, whose launches are mostly ramp-up (one token
    // through 32 8B-class layers, 128 launches of 4-117 MB: 1.59 -> 1.85 ms),
    // so it is on only when a CTA streams at least 1 MiB of M.
    const bool prefetch = args.base[count] / grid >= (1LL << 20);
    const auto kern = prefetch ? k_gemv_multi<2, 4, true> : k_gemv_multi<2, 4, false>;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid, 1, 1);
    cfg.blockDim = dim3(kMultiThreads, 1, 1);
    cfg.dynamicSmemBytes = (size_t)4 * kmax;
    cfg.stream = s;
    cudaLaunchAttribute attrs[1];
    attrs[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attrs[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attrs;
    cfg.numAttrs = 1;
    return counted_launch(cudaLaunchKernelEx(&cfg, kern, args));
}

template <int ROWS, int UNROLL, bool kVec>
cudaError_t run_gemv(const int8_t *W, size_t ldw, int m, int K, const uint32_t *xhat, uint32_t *y,
                     bool accumulate, cudaStream_t s) {
    const int nchunks = (K + 15) / 16;
    const size_t smem = (size_t)nchunks * 16 * 4;
    auto kern = k_gemv<ROWS, UNROLL, kVec>;
    // set once (outside any stream capture that a later call might be part of)
    const cudaError_t attr = func_attr((const void *)kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       kGemvMaxK * 4);
    if (attr != cudaSuccess) return attr;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int ngroups = (m + ROWS - 1) / ROWS;
    const int grid = ngroups < sms ? ngroups : sms;
    kern<<<grid, kGemvThreads, smem, s>>>(W, ldw, m, K, xhat, y, accumulate); note_launch();
    return cudaGetLastError();
}

}  // namespace

bool multi_eligible(const MvmJob &j) {
    return j.K % 16 == 0 && j.ldw % 16 == 0 && (reinterpret_cast<uintptr_t>(j.W) & 15u) == 0 &&
           (reinterpret_cast<uintptr_t>(j.xhat) & 15u) == 0;
}

cudaError_t launch_gemv_multi(const MvmJob *jobs, int count, cudaStream_t s) {
    // Jobs with K beyond one shared-memory segment are split into K segments;
    // segment k of every job goes into launch k, later launches accumulate.
    std::vector<MvmJob> seg;
    for (int k0 = 0;; k0 += kMultiMaxK) {
        seg.clear();
        for (int j = 0; j < count; ++j) {
            if (jobs[j].K <= k0) continue;
            MvmJob t = jobs[j];
            t.W = jobs[j].W + k0;
            t.xhat = jobs[j].xhat + k0;
            t.K = jobs[j].K - k0 < kMultiMaxK ? jobs[j].K - k0 : kMultiMaxK;
            t.accumulate = k0 > 0 ? 1 : jobs[j].accumulate;
            seg.push_back(t);
        }
        if (seg.empty()) return cudaSuccess;
        for (size_t a = 0; a < seg.size(); a += kMultiMaxJobs) {
            const int n = (int)std::min(seg.size() - a, (size_t)kMultiMaxJobs);
            cudaError_t e = run_gemv_multi(seg.data() + a, n, s);
            if (e != cudaSuccess) return e;
        }
    }
}

cudaError_t launch_gemv(const int8_t *W, int m, int K, const uint32_t *xhat, uint32_t *y,
                        uint32_t *err, cudaStream_t s) {
    (void)err;
    if (m <= 0 || K <= 0) return cudaSuccess;
    MvmJob j{W, xhat, y, m, K, (size_t)K, 0};
    if (multi_eligible(j)) return launch_gemv_multi(&j, 1, s);
    for (int k0 = 0; k0 < K; k0 += kGemvMaxK) {
        const int kl = K - k0 < kGemvMaxK ? K - k0 : kGemvMaxK;
        cudaError_t e = run_gemv<2, 2, false>(W + k0, (size_t)K, m, kl, xhat + k0, y, k0 > 0, s);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace pv
