// Host-side launchers of the pvMVMD kernels (internal to the library).
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

#include "pvmvmd.h"

namespace pv {

// Positions per tile of the single-lane syndrome scan.
constexpr int kScanThreads = 256;
constexpr int kScanItems = 8;
constexpr int kScanTile = kScanThreads * kScanItems;

__host__ __device__ inline uint32_t scan_tiles(uint32_t N) { return (N + kScanTile - 1) / kScanTile; }

// Status words a syndrome scan over `count` vectors of length N needs
// (word 0 is the tile ticket).
inline size_t scan_status_words(uint32_t N, uint32_t count) {
    return 1 + (size_t)count * scan_tiles(N);
}

// Sample `count` vectors of E_t^N: vector j uses index idx0 + j, reading
// nonces (tag, 2*idx) and (tag, 2*idx + 1).  out: [count][2t] (ascending
// support, then values).  Also zeroes clear[0 .. clear_words) for the scan
// that follows in the same stream.
cudaError_t launch_sample_sparse(const pvmvmd_key &key, uint32_t tag, uint64_t idx0, uint32_t N,
                                 uint32_t t, uint32_t count, uint32_t *out,
                                 unsigned long long *clear, size_t clear_words, cudaStream_t s);

// Syndrome scan part of x' = G e for sparse e (App. B, syndrome direction):
// c_i = v2[pi2^-1(i)] * (A e)_{pi2^-1(i)}, d = A c (suffix sums),
// F_i = v1_i * d_i.  sparse: [count][2t]; F: [count][N].
cudaError_t launch_syndrome_scan(const uint32_t *pi2inv, const uint32_t *v2p, const uint32_t *v1,
                                 uint32_t N, const uint32_t *sparse, uint32_t t, uint32_t count,
                                 uint32_t *F, unsigned long long *status, uint32_t *err,
                                 cudaStream_t s);

// Cluster spread of the fused syndrome (how far a small batch's clusters
// grow): encodes of a few vectors, and the few shared challenges of a
// verification, each measured best at a different setting.  The challenges
// of a large batch run beside a large decrypt and keep their clusters
// small; those of a small batch, and those of boost mode (no decrypt of
// P^T rows beside them), are the decode's critical path.
constexpr int kSpreadEncode = 4;
constexpr int kSpreadChallenge = 16;
constexpr int kSpreadChallengeSmallBatch = 4;
constexpr int kChallengeLargeBatch = 32;

// Fused syndrome for `count` freshly sampled sparse vectors (as
// launch_sample_sparse, then out = addend + G e) in one launch with the
// intermediate in cluster shared memory.  sparse_out: [count][2t];
// out (and addend, may alias): [count][n].  cudaErrorNotSupported when N is
// too long for one cluster (use the three-kernel path).
bool syndrome_fused_plan(uint32_t N, uint32_t t, int *C, uint32_t *slice, size_t *smem);
// Tables: pi2inv, v2p = v2 o pi2^-1, v1 (cluster form); pi2, v2m = v2 R,
// v1pm = (v1 o pi1^-1) R (single-CTA form, Montgomery-scaled, R = 2^32).
// pdl: launch with programmatic stream serialisation.  The kernel reads
// nothing but the key and the tables before griddepcontrol.wait, so its
// sampling and scans overlap the kernel before it; st, out and addend are
// touched only after the wait.
cudaError_t launch_syndrome_fused(const pvmvmd_key &key, uint32_t tag, uint64_t idx0, uint32_t N,
                                  uint32_t t, uint32_t count, const uint32_t *pi2inv,
                                  const uint32_t *v2p, const uint32_t *v1, const uint32_t *pi1inv,
                                  const uint32_t *pi2, const uint32_t *v2m, const uint32_t *v1pm,
                                  uint32_t n, uint32_t r, uint32_t *sparse_out,
                                  const uint32_t *addend, uint32_t *out, cudaStream_t s,
                                  bool pdl = false, int spread = kSpreadChallenge);

// Lane-parallel syndrome for L vectors (vector b uses index idx0 + b, as
// launch_sample_sparse): sparse_out [L][2t] as there, S lane_state_words(t,
// L) words (suffix sums of the values, then a bucket index into the sorted
// supports), C [N][L rounded up to 4] the intermediate (16-byte
// aligned), aux lane_aux_words(N, L) words (16-byte aligned); out = addend +
// G e with out, addend [L][n] (addend may be null or alias out).  Tables:
// pi2, v2m = v2 R and v1m = v1 R (Montgomery, R = 2^32), pi1inv.
size_t lane_state_words(uint32_t t, uint32_t L);
size_t lane_aux_words(uint32_t N, uint32_t L);
cudaError_t launch_lane_syndrome(const pvmvmd_key &key, uint32_t tag, uint64_t idx0, uint32_t N,
                                 uint32_t t, uint32_t L, const uint32_t *pi2, const uint32_t *v2m,
                                 const uint32_t *v1m, const uint32_t *pi1inv, uint32_t n, uint32_t r,
                                 uint32_t *sparse_out, uint32_t *S, uint32_t *C, uint32_t *aux,
                                 const uint32_t *addend, uint32_t *out, cudaStream_t s);

// Gather part: out_j = addend_j + sum_{c<r} F[pi1^-1(r j + c)], j < n
// (addend may be null; out may alias addend).
cudaError_t launch_syndrome_gather(const uint32_t *pi1inv, uint32_t n, uint32_t r,
                                   const uint32_t *F, uint32_t N, const uint32_t *addend,
                                   uint32_t *out, uint32_t count, cudaStream_t s);

// Every kernel launch site calls note_launch() (or wraps a cudaLaunchKernelEx
// in counted_launch), so that pvmvmd_kernel_launches counts what the library
// enqueued.
void note_launch();
inline cudaError_t counted_launch(cudaError_t e) {
    if (e == cudaSuccess) note_launch();
    return e;
}

// One accumulate stage of the encoding G^T w over L lanes (App. B, encoding
// direction): Y[j][l] = sum_{j' <= j} vscale[j'] * X[perm[j'] / div][l] for
// j < N, with vscale_m = vscale R mod q (Montgomery form, R = 2^32).  X is
// int8 (lifted to F_q) when x_is_i8, else uint32.  Scratch: `status` holds
// encode_scan_status_words(N, L) 64-bit words and `ticket` one 32-bit word,
// all zero at launch (encode_scan_clear).
constexpr int kEncTile = 32;
size_t encode_scan_status_words(uint32_t N, uint32_t L);
cudaError_t encode_scan_clear(unsigned long long *status, uint32_t *ticket, uint32_t N, uint32_t L,
                              cudaStream_t s);
cudaError_t launch_encode_scan(const void *X, bool x_is_i8, size_t ldx, const uint32_t *perm,
                               uint32_t div, const uint32_t *vscale_m, uint32_t N, uint32_t L,
                               uint32_t *Y, size_t ldy, unsigned long long *status, uint32_t *ticket,
                               uint32_t *err, cudaStream_t s);

// int8 transpose: out[c][r] = in[r][c] for an R x C matrix.
cudaError_t launch_transpose_i8(const int8_t *in, int R, int C, int8_t *out, cudaStream_t s);

// One independent batch-1 product y = M x_hat over F_q (M row stride ldw).
struct MvmJob {
    const int8_t *W;
    const uint32_t *xhat;
    uint32_t *y;
    int m, K;
    size_t ldw;
    int accumulate;  // y += M x_hat instead of y = M x_hat
};
constexpr int kMultiMaxJobs = 256;  // jobs per grouped launch
constexpr int kMultiMaxK = 16384;   // K per grouped launch (longer K is segmented)

// Y_hat = M X_hat for a few vectors (2 <= B <= 16): one pass over M per group
// of four vectors.  Needs K % 16 == 0 and 16-byte aligned W and X_hat.
cudaError_t launch_gemv_small_batch(const int8_t *W, int m, int K, const uint32_t *Xhat, int B,
                                    uint32_t *Yhat, cudaStream_t s);

// Eligible for the grouped kernel: K % 16 == 0 and 16-byte aligned rows.
bool multi_eligible(const MvmJob &j);
// Any number of eligible jobs, in as few launches as K allows.
cudaError_t launch_gemv_multi(const MvmJob *jobs, int count, cudaStream_t s);

// Batch-1 field GEMV y = M x_hat over F_q.
cudaError_t launch_gemv(const int8_t *W, int m, int K, const uint32_t *xhat, uint32_t *y,
                        uint32_t *err, cudaStream_t s);

// Batched product Y_hat[b] = M x_hat[b] over F_q on the tensor cores.
cudaError_t launch_batched(const int8_t *W, int m, int K, const uint32_t *Xhat, int B,
                           uint32_t *Yhat, uint32_t *err, cudaStream_t s);

// Several independent batched products in one persistent tensor-core launch
// (jobs with K % 16 == 0 and 16-byte aligned W; outputs must not overlap).
struct BatchJob {
    const int8_t *W;
    const uint32_t *Xhat;
    uint32_t *Yhat;
    int m, K, B;
};
bool batched_grouped_eligible(const int8_t *W, int m, int K, int B);
cudaError_t launch_batched_grouped(const BatchJob *jobs, int count, uint32_t *err, cudaStream_t s);

// Grow-only scratch of at least `need` bytes for `purpose` on the current
// device, one buffer per stream (see scratch.cu).
enum ScratchPurpose { kScratchDigitTiles = 0, kScratchDigitPlanes = 1 };
cudaError_t stream_scratch(int purpose, size_t need, cudaStream_t s, void **out);

// cudaFuncSetAttribute for the current device, done once per (kernel,
// attribute, device): function attributes belong to each device's instance
// of the kernel.
cudaError_t func_attr(const void *fn, cudaFuncAttribute attr, int value);

// The library's device error word on the current device (null on failure).
uint32_t *library_error_word();

// The failure-path test hook (pvmvmd_debug_expire_wait): which bounded wait
// to make expire, where, and the shortened limit.  site 0 = off.
struct DebugWait {
    int site = 0;
    uint32_t index = 0;
    uint64_t limit = 0;
};
DebugWait debug_wait();

// Verify part 1: u[q][k] = sum_j e_{q,j} Q[supp_{q,j}][k] (e_q^T Q).
cudaError_t launch_verify_u(const uint32_t *Qm, int K, const uint32_t *chal, uint32_t t_y,
                            uint32_t ell, uint32_t *u, cudaStream_t s);

// Decrypt: Y[b] = Y_hat[b] - P e_x,b for B vectors (st [B][2t_x], support
// indices below Nx; others read row 0); with
// mask non-null (boost mode) Y = Y_hat - mask, mask [B][m] = P e_x per
// vector, and st is not read.  Y may alias Y_hat.
cudaError_t launch_decrypt(const uint32_t *PT, int m, const uint32_t *st, uint32_t t_x, uint32_t Nx,
                           const uint32_t *Yhat, int B, uint32_t *Y, cudaStream_t s,
                           const uint32_t *mask = nullptr);
// Verify: accept[b] = AND_q (u_q . Xhat[b] == g_q . Yhat[b]) for the ell
// challenges' u (ell x K) and g (ell x m).
cudaError_t launch_check(const uint32_t *Xhat, int K, const uint32_t *Yhat, int m, const uint32_t *g,
                         const uint32_t *u, uint32_t ell, int B, int32_t *accept, cudaStream_t s);

// out = a + b over F_q (n elements; out may alias a or b).
cudaError_t launch_field_add(const uint32_t *a, const uint32_t *b, size_t n, uint32_t *out,
                             cudaStream_t s);

// Output masks out[b] = P e_x,b (m values) from st [B][2t_x].
cudaError_t launch_output_mask(const uint32_t *PT, int m, const uint32_t *st, uint32_t t_x, int B,
                               uint32_t *out, cudaStream_t s);

// out (C x R) = in (R x C) transposed, uint32.
cudaError_t launch_transpose_u32(const uint32_t *in, int R, int C, uint32_t *out, cudaStream_t s);

// Protocol 2's client checks; accept = 1 iff every check holds.  QauxT
// [N'][N], chal [ell][2t] and chal2 [ell'][2t'] (ascending support, then
// values), u [ell][Bn] the server's projections, R [ell'][Bn] = G' e',
// X [B][n] the claims' inputs, Z [N][B] = G^T y_b.
cudaError_t launch_bv_checks(const uint32_t *QauxT, int N, int Bn, int n, int B, const uint32_t *chal,
                             uint32_t t, uint32_t ell, const uint32_t *chal2, uint32_t t2, uint32_t ell2,
                             const uint32_t *u, const uint32_t *R, const uint32_t *X, const uint32_t *Z,
                             int32_t *accept, cudaStream_t s);

// 16-bit weights: W = 256 hi + lo (int8 planes, w in [-32768, 32639]);
// W lifted to F_q; y = 256 y + ylo over F_q.
cudaError_t launch_split_i16(const int16_t *W, size_t n, int8_t *hi, int8_t *lo, cudaStream_t s);
cudaError_t launch_lift_i16(const int16_t *W, size_t n, uint32_t *out, cudaStream_t s);
cudaError_t launch_combine_256(uint32_t *y, const uint32_t *ylo, size_t n, cudaStream_t s);

}  // namespace pv
