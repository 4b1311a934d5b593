// Server product for a few vectors (2 <= B <= 16; Sec. 6.1): Y_hat = M X_hat
// over F_q with one pass over M per group of four vectors.  The arithmetic
// is the batch-1 GEMV's (four signed base-256 digit planes of x_hat, dp4a,
// exact int32 sums, one reduction mod q per output); each 16 bytes of M now
// feed four vectors' planes.
#include <algorithm>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "launch.h"

namespace pv {
namespace {

constexpr int kMultiThreads = 256;
constexpr int kMultiWarps = kMultiThreads / 32;

__device__ __forceinline__ uint4 ldg_stream(const void *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// Sum of v[lane] over the 32 lanes for V = 32 entries per lane: after the
// call lane e holds the total of entry e (a transposed butterfly).
template <int V>
__device__ __forceinline__ int transposed_reduce(int (&v)[V], int lane) {
    static_assert(V == 32, "one entry per lane");
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
    return v[0];
}

// ---------------------------------------------------------------------------
// Small batches (2 <= B <= 16): one pass over M serves up to four vectors.
// The digit planes of the four vectors' x_hat segment sit side by side in
// shared memory; every 16 bytes of M feed 16 dp4a per vector, so M is read
// once per group of four vectors instead of once per vector, and the
// tensor-core product's 64-vector tiles are not wasted on a few vectors.
// Same row split and streaming as the grouped batch-1 kernel: the bytes of
// all jobs are split evenly over 2 CTAs per SM (whole rows), warps stream
// row pairs with the next loads issued before the current arithmetic.
// ---------------------------------------------------------------------------
constexpr int kNbVec = 4;          // vectors per pass
constexpr int kNbMaxK = 6144;      // K per pass (4 planes x 4 vectors x K bytes)
constexpr int kNbMaxJobs = 32;
// Each of the 16 plane rows in shared memory is kNbMaxK bytes apart whatever
// K is, so the 16 row offsets of the inner loop are compile-time constants
// (immediate offsets of one address per chunk).
constexpr int kNbStride = kNbMaxK / 16;  // 16-byte chunks per plane row
constexpr int kNbSmem = 4 * kNbVec * kNbMaxK;

struct NbJob {
    const int8_t *W;
    const uint32_t *planes;  // row (p, v) of the segment at planes + (p * kNbVec + v) * ldp
    uint32_t *y;             // vector v at y + v * ldy
    int m, K, nb, accumulate;
    size_t ldw, ldp, ldy;    // ldp in 32-bit words
};
struct NbArgs {
    int count;
    long long base[kNbMaxJobs + 1];
    NbJob job[kNbMaxJobs];
};

// Digit planes of the batch, once per call: planes[j][p][v][k] (int8) is
// digit p of centred x_hat[4j + v][k]; vectors past B are zero.  One thread
// per four consecutive K-elements of one vector.
__global__ void __launch_bounds__(256) k_nb_planes(const uint32_t *__restrict__ Xhat, int B, int K, int Bp,
                                                  uint32_t *__restrict__ planes) {
    asm volatile("griddepcontrol.wait;" ::: "memory");  // x_hat comes from the kernel before
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const size_t gid = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const size_t per_vec = (size_t)K / 4;
    if (gid >= (size_t)Bp * per_vec) return;
    const int b = (int)(gid / per_vec), q4 = (int)(gid % per_vec);
    uint32_t p[4] = {0u, 0u, 0u, 0u};
    if (b < B) {
        const uint4 xv = __ldg(reinterpret_cast<const uint4 *>(Xhat + (size_t)b * K) + q4);
        const uint32_t xs[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            int d0, d1, d2, d3;
            limb_split(xs[e], d0, d1, d2, d3);
            p[0] |= (uint32_t)(d0 & 0xff) << (8 * e);
            p[1] |= (uint32_t)(d1 & 0xff) << (8 * e);
            p[2] |= (uint32_t)(d2 & 0xff) << (8 * e);
            p[3] |= (uint32_t)(d3 & 0xff) << (8 * e);
        }
    }
    const int j = b / kNbVec, v = b % kNbVec;
    uint32_t *dst = planes + (size_t)j * 4 * kNbVec * per_vec;
#pragma unroll
    for (int d = 0; d < 4; ++d) dst[((size_t)d * kNbVec + v) * per_vec + q4] = p[d];
}

template <int ROWS, int UNROLL>
__global__ void __launch_bounds__(kMultiThreads, 2) k_gemv_nb(const __grid_constant__ NbArgs args) {
    extern __shared__ uint4 s_planes[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr int V = ROWS * 4 * kNbVec;
    static_assert(V == 32, "ROWS * 4 planes * 4 vectors must be one entry per lane");
    const long long total = args.base[args.count];
    const long long lo = total * blockIdx.x / gridDim.x;
    const long long hi = total * (blockIdx.x + 1) / gridDim.x;

    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    // The first loads of M go out before griddepcontrol.wait (M is the
    // server's weight matrix, never written by a kernel of the chain); the
    // planes and y_hat are touched only after it.
    bool waited = false;

    for (int j = 0; j < args.count; ++j) {
        const long long b0 = args.base[j], b1 = args.base[j + 1];
        if (b1 <= lo || b0 >= hi) continue;
        const NbJob &job = args.job[j];
        const int K = job.K, m = job.m, nchunks = K / 16;
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
        // planes: row p * kNbVec + v holds plane p of vector v, copied from
        // the planes the call built once; rows of vectors past nb are zero
        for (int c = tid; c < nchunks; c += kMultiThreads) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                uint4 t[8];
#pragma unroll
                for (int r = 0; r < 8; ++r)
                    t[r] = __ldg(reinterpret_cast<const uint4 *>(job.planes + (size_t)(8 * h + r) * job.ldp) + c);
#pragma unroll
                for (int r = 0; r < 8; ++r) s_planes[(8 * h + r) * kNbStride + c] = t[r];
            }
        }
        __syncthreads();

        for (; g < ngroups; g += kMultiWarps) {
            int acc[ROWS][kNbVec][4];
#pragma unroll
            for (int r = 0; r < ROWS; ++r)
#pragma unroll
                for (int v = 0; v < kNbVec; ++v) acc[r][v][0] = acc[r][v][1] = acc[r][v][2] = acc[r][v][3] = 0;
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
#pragma unroll
                        for (int v = 0; v < kNbVec; ++v) {
                            uint4 l[4];
#pragma unroll
                            for (int p = 0; p < 4; ++p) l[p] = s_planes[(p * kNbVec + v) * kNbStride + cc];
#pragma unroll
                            for (int r = 0; r < ROWS; ++r) {
                                const uint4 w = cur[u][r];
#pragma unroll
                                for (int p = 0; p < 4; ++p) {
                                    acc[r][v][p] = __dp4a((int)w.x, (int)l[p].x, acc[r][v][p]);
                                    acc[r][v][p] = __dp4a((int)w.y, (int)l[p].y, acc[r][v][p]);
                                    acc[r][v][p] = __dp4a((int)w.z, (int)l[p].z, acc[r][v][p]);
                                    acc[r][v][p] = __dp4a((int)w.w, (int)l[p].w, acc[r][v][p]);
                                }
                            }
                        }
                    }
                }
            }
            // entry e = (r * kNbVec + v) * 4 + p: lane e ends with its total
            int vals[V];
#pragma unroll
            for (int r = 0; r < ROWS; ++r)
#pragma unroll
                for (int v = 0; v < kNbVec; ++v)
#pragma unroll
                    for (int p = 0; p < 4; ++p) vals[(r * kNbVec + v) * 4 + p] = acc[r][v][p];
            const int tot = transposed_reduce<V>(vals, lane);
            const int a1 = __shfl_down_sync(kFull, tot, 1);
            const int a2 = __shfl_down_sync(kFull, tot, 2);
            const int a3 = __shfl_down_sync(kFull, tot, 3);
            if ((lane & 3) == 0) {
                const int v = (lane >> 2) % kNbVec, r = (lane >> 2) / kNbVec;
                const int row = row_a + g * ROWS + r;
                if (row < row_b && v < job.nb) {
                    const int64_t sum = (int64_t)tot + ((int64_t)a1 << 8) + ((int64_t)a2 << 16) +
                                        ((int64_t)a3 << 24);
                    const uint32_t part = fred_signed(sum);
                    uint32_t *yp = job.y + (size_t)v * job.ldy + row;
                    *yp = job.accumulate ? fadd(*yp, part) : part;
                }
            }
        }
    }
    // a CTA with no rows still waits, so that the kernel completes only
    // after the one before it (dependents rely on that order)
    if (!waited) asm volatile("griddepcontrol.wait;" ::: "memory");
}

cudaError_t run_gemv_nb(const NbJob *jobs, int count, cudaStream_t s) {
    static NbArgs args;  // host staging of the kernel parameters (copied at launch)
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    args.count = count;
    args.base[0] = 0;
    long long rows = 0;
    for (int j = 0; j < count; ++j) {
        args.job[j] = jobs[j];
        args.base[j + 1] = args.base[j] + (long long)jobs[j].m * jobs[j].K;
        rows += jobs[j].m;
    }
    if (rows == 0) return cudaSuccess;
    const cudaError_t attr =
        func_attr((const void *)k_gemv_nb<2, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, kNbSmem);
    if (attr != cudaSuccess) return attr;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    long long grid = 2LL * sms;
    if (grid > rows) grid = rows;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid, 1, 1);
    cfg.blockDim = dim3(kMultiThreads, 1, 1);
    cfg.dynamicSmemBytes = kNbSmem;
    cfg.stream = s;
    cudaLaunchAttribute attrs[1];
    attrs[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attrs[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attrs;
    cfg.numAttrs = 1;
    return counted_launch(cudaLaunchKernelEx(&cfg, k_gemv_nb<2, 2>, args));
}

}  // namespace

cudaError_t launch_gemv_small_batch(const int8_t *W, int m, int K, const uint32_t *Xhat, int B,
                                    uint32_t *Yhat, cudaStream_t s) {
    if (m <= 0 || K <= 0 || B <= 0) return cudaSuccess;
    // digit planes of all vectors once: [job][plane][vector][K] bytes
    const int Bp = (B + kNbVec - 1) / kNbVec * kNbVec;
    const size_t row_words = (size_t)K / 4, job_words = 4 * kNbVec * row_words;
    void *pbuf = nullptr;
    cudaError_t e = stream_scratch(kScratchDigitPlanes, (size_t)Bp / kNbVec * job_words * sizeof(uint32_t), s, &pbuf);
    if (e != cudaSuccess) return e;
    uint32_t *planes = static_cast<uint32_t *>(pbuf);
    {
        const size_t threads = (size_t)Bp * row_words;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)((threads + 255) / 256), 1, 1);
        cfg.blockDim = dim3(256, 1, 1);
        cfg.stream = s;
        cudaLaunchAttribute attrs[1];
        attrs[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attrs[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attrs;
        cfg.numAttrs = 1;
        if ((e = counted_launch(cudaLaunchKernelEx(&cfg, k_nb_planes, Xhat, B, K, Bp, planes))) != cudaSuccess) return e;
    }
    // groups of four vectors; K in segments whose planes fit shared memory,
    // later segments accumulating
    std::vector<NbJob> jobs;
    for (int k0 = 0; k0 < K; k0 += kNbMaxK) {
        jobs.clear();
        const int kl = K - k0 < kNbMaxK ? K - k0 : kNbMaxK;
        for (int b0 = 0; b0 < B; b0 += kNbVec) {
            NbJob j;
            j.W = W + k0;
            j.planes = planes + (size_t)(b0 / kNbVec) * job_words + (size_t)k0 / 4;
            j.y = Yhat + (size_t)b0 * m;
            j.m = m;
            j.K = kl;
            j.nb = B - b0 < kNbVec ? B - b0 : kNbVec;
            j.accumulate = k0 > 0;
            j.ldw = (size_t)K;
            j.ldp = row_words;
            j.ldy = (size_t)m;
            jobs.push_back(j);
        }
        for (size_t a = 0; a < jobs.size(); a += kNbMaxJobs) {
            const int n = (int)std::min(jobs.size() - a, (size_t)kNbMaxJobs);
            e = run_gemv_nb(jobs.data() + a, n, s);
            if (e != cudaSuccess) return e;
        }
    }
    return cudaSuccess;
}

}  // namespace pv
