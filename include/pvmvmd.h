/*
 * pvmvmd.h — C ABI of the GB300 (sm_103a) pvMVMD library.
 *
 * The calls follow Protocol 3 (Pi_pvMVMD) of the Maverick paper
 * (arXiv 2609.10264, Sec. 6.1) and Def. 4.2's algorithm split:
 *   pvmvmd_preprocess      Preprocess(M) -> pp = (G_x, G_y, P, Q, t_x, t_y, ell)
 *   pvmvmd_encode          Encrypt(pp, x) -> (x_hat, st)
 *   pvmvmd_server_mvm      the server's y_hat = M x_hat over F_q
 *   pvmvmd_decode_verify   Verify(pp, x_hat, y_hat) and Decrypt(pp, st, y_hat)
 * The codes are the RAA codes of App. B, G = R Pi1 V1 A Pi2 V2 A, with the
 * parameters of Sec. 7.1 by default.
 *
 * Conventions shared by every call
 *  - Field: BabyBear, q = 15 * 2^27 + 1 = 2013265921 (Sec. 7.1).  Every field
 *    element crossing the ABI is a uint32 in canonical form [0, q).  Inputs
 *    outside [0, q) give unspecified (but memory-safe) results.
 *  - The public matrix M is int8, row-major m x K, embedded in F_q by
 *    w -> w mod q (Sec. 7.2.1 embeds signed quantised weights the same way).
 *  - A batch of B vectors of length L is stored vector after vector
 *    ("B x L row-major"): vector b occupies elements [b*L, (b+1)*L).
 *  - Pointers named *_dev are CUDA device pointers on the current device;
 *    the caller owns them.  The library owns only what a context holds.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Every call only enqueues work on that stream and returns;
 *    results are valid once the stream has been synchronised.  Calls that use
 *    one context must be ordered on one stream (a context's internal scratch
 *    is shared by its calls), with one exception: an encode
 *    (pvmvmd_encode, pvmvmd_boost_prepare) and a decode
 *    (pvmvmd_decode_verify, pvmvmd_boost_decode_verify) share no scratch, so
 *    the encode of one batch may run on another stream while an earlier
 *    batch is decoded.
 *  - Return value: PVMVMD_OK (0) or a negative PVMVMD_E_* status.  Nothing
 *    throws across the ABI.  A device-side bounded wait that expires is
 *    reported later by pvmvmd_device_status.
 *  - Randomness: a pvmvmd_key is a 256-bit ChaCha20 key (RFC 8439); each
 *    sampled object reads its own keystream, selected by the nonce
 *    (domain tag, index).  Encode keys must never be reused: masks derived
 *    from a reused key repeat, which voids privacy.
 */
#ifndef PVMVMD_H
#define PVMVMD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define PVMVMD_Q 2013265921u

/* Largest K for which the server product's per-digit int32 sums cannot
 * overflow for any int8 weight: 128 * 128 * K < 2^31. */
#define PVMVMD_MAX_K 131071

/* Largest sparsity accepted for t_x and t_y. */
#define PVMVMD_MAX_T 4096

enum {
    PVMVMD_OK = 0,
    PVMVMD_E_ARG = -1,            /* null pointer or invalid argument          */
    PVMVMD_E_SHAPE = -2,          /* m, K or B outside the supported range      */
    PVMVMD_E_PARAM = -3,          /* parameters inconsistent (e.g. t > N)       */
    PVMVMD_E_CUDA = -4,           /* a CUDA runtime call or launch failed       */
    PVMVMD_E_NOMEM = -5,          /* device or host allocation failed           */
    PVMVMD_E_DEVICE_TIMEOUT = -6, /* a bounded device-side wait expired         */
    PVMVMD_E_NODEVICE = -7        /* no sm_103 device is current                */
};

/* 256-bit ChaCha20 key, eight little-endian 32-bit words. */
typedef struct { uint32_t k[8]; } pvmvmd_key;

/* Protocol parameters.  A zero field selects the paper's value. */
typedef struct {
    int lambda;        /* computational security parameter; 0 -> 128 (Sec. 7.1)        */
    int kappa;         /* statistical security parameter; 0 -> 40 (Sec. 7.1)           */
    int rate;          /* N / dimension of both RAA codes; 0 -> 8 (rate 1/8, Sec. 7.1) */
    double delta;      /* target relative distance; 0 -> 0.5 (Sec. 7.1)                */
    int t_x;           /* mask sparsity; 0 -> Eq. (1), ceil(ln2 (lambda - log2 N_x)/delta) */
    int t_y;           /* challenge sparsity; 0 -> Thm 5.2 by its proof's two cases
                          (31 for BabyBear with kappa = 40, delta = 1/2, as Sec. 7.1 uses) */
    int ell;           /* challenge repetitions; 0 -> Thm 5.2 (2 with Sec. 7.1's values) */
    int scratch_batch; /* vectors per internal encode chunk; 0 -> 64 (memory knob only) */
} pvmvmd_params;

typedef struct pvmvmd_ctx pvmvmd_ctx;

/* Read-only view of a context's public parameters pp (Protocol 3).  All
 * arrays are device memory owned by the context.  Permutations follow App. B:
 * pi[j] = pi(j), and Pi_{i,j} = 1 iff pi(j) = i. */
typedef struct {
    int m, K;                 /* matrix shape                                   */
    int rate, N_x, N_y;       /* N_x = rate*K (privacy code), N_y = rate*m (verification code) */
    int t_x, t_y, ell;
    const uint32_t *gx_pi1, *gx_pi2, *gx_v1, *gx_v2; /* G_x, each length N_x    */
    const uint32_t *gy_pi1, *gy_pi2, *gy_v1, *gy_v2; /* G_y, each length N_y    */
    const uint32_t *PT;       /* P^T = (M G_x)^T, row-major N_x x m              */
    const uint32_t *Q;        /* Q = G_y^T M, row-major N_y x K                  */
} pvmvmd_ctx_view;

/* Fill every zero field of *in with the paper's default for an m x K matrix
 * (Eq. 1, Thm 5.2, Sec. 7.1) and write the result to *out.  Host only; needs
 * no GPU.  Returns PVMVMD_E_PARAM if the resolved t_x > rate*K,
 * t_y > rate*m, either t exceeds PVMVMD_MAX_T, or a field is negative. */
int pvmvmd_params_resolve(const pvmvmd_params *in, int m, int K, pvmvmd_params *out);

/* Preprocess(M) (Protocol 3; P and Q as in Sec. 6.3): samples G_x (dimension
 * K) and G_y (dimension m) from `key`, computes P^T = G_x^T M^T (m encodings of
 * the rows of M) and Q = G_y^T M (K encodings of its columns) on the device,
 * and returns a context owning them.  W_dev: int8 m x K row-major; W need
 * not stay alive afterwards.  params may be NULL (all defaults).
 * 1 <= m, 1 <= K <= PVMVMD_MAX_K.  Allocates about 8*rate*m*K bytes of device
 * memory plus code tables and scratch; the call synchronises `stream` before
 * returning.  The context also owns one CUDA stream, created at the device's
 * highest stream priority, on which pvmvmd_decode_verify runs its short
 * verification kernels beside the decrypt.  On error *out is NULL. */
int pvmvmd_preprocess(const int8_t *W_dev, int m, int K, const pvmvmd_params *params,
                      const pvmvmd_key *key, void *stream, pvmvmd_ctx **out);

/* Bytes of the private state st for B vectors: B * 2 * t_x uint32 (for
 * vector b, its mask's support in ascending order, then the matching values). */
int pvmvmd_state_size(const pvmvmd_ctx *ctx, int B, size_t *bytes);

/* Encrypt (Protocol 3): for each of the B vectors x_b (X_dev, B x K), sample
 * e_x <- E_{t_x}^{N_x} from `key` (vector b reads nonce (9, 2b) for its support
 * and (9, 2b+1) for its values), write x_hat_b = x_b + G_x e_x to Xhat_dev
 * (B x K) and st_b = e_x to st_dev (pvmvmd_state_size bytes).  B >= 1.
 * X_dev and Xhat_dev may alias. */
int pvmvmd_encode(pvmvmd_ctx *ctx, const uint32_t *X_dev, int B, const pvmvmd_key *key,
                  uint32_t *Xhat_dev, void *st_dev, void *stream);

/* The server's product Y_hat = M X_hat over F_q (Sec. 6.1: the server's whole
 * online work).  W_dev int8 m x K row-major, Xhat_dev B x K, Yhat_dev B x m.
 * Needs no context and no secret.  B == 1 runs the bandwidth-bound GEMV;
 * 2 <= B <= 16 (K a multiple of 16, 16-byte aligned W and Xhat) a GEMV that
 * reads M once per four vectors, or, for B >= 8 and m K B >= 2^27, the
 * tensor-core product with 16-vector tiles; larger B the byte-limb
 * tensor-core product.
 * 1 <= K <= PVMVMD_MAX_K.  The batch-1 GEMV and the 2 <= B <= 16 GEMV may
 * start reading M while the kernel before it on the stream finishes, when
 * that kernel signals its
 * dependents early (programmatic dependent launch); such a kernel must not
 * write M.  Kernels that do not use programmatic dependent launch, and all
 * of this library's kernels, are safe.  The B > 1 paths keep their digit
 * operand in library scratch held per stream: calls on different streams
 * may run concurrently, and a buffer grows (with a synchronisation of the
 * stream) only when a call needs more than any earlier call on that stream,
 * which must not happen while the stream is being captured. */
int pvmvmd_server_mvm(const int8_t *W_dev, int m, int K, const uint32_t *Xhat_dev, int B,
                      uint32_t *Yhat_dev, void *stream);

/* One request of pvmvmd_server_mvm_multi: yhat = W xhat over F_q. */
typedef struct {
    const int8_t *W_dev;      /* int8 m x K row-major                       */
    const uint32_t *xhat_dev; /* K field elements                           */
    uint32_t *yhat_dev;       /* m field elements (output)                  */
    int m, K;
} pvmvmd_mvm_job;

/* The server's products for `count` independent batch-1 requests (Sec. 6.1:
 * the server's online work is one product per masked vector), in as few
 * launches as possible: jobs[i].yhat_dev = jobs[i].W_dev * jobs[i].xhat_dev
 * over F_q.  Requests may use different matrices and shapes; each matrix is
 * streamed once per request (no reuse across requests).  Results equal
 * `count` calls of pvmvmd_server_mvm with B = 1.  `jobs` is a host array that
 * may be freed on return; outputs must not overlap any input or each other.
 * 1 <= count, each 1 <= K <= PVMVMD_MAX_K, 1 <= m. */
int pvmvmd_server_mvm_multi(const pvmvmd_mvm_job *jobs, int count, void *stream);

/* One product of pvmvmd_server_mvm_grouped: Yhat = W Xhat over F_q for a
 * batch of B vectors (Xhat_dev B x K, Yhat_dev B x m). */
typedef struct {
    const int8_t *W_dev;      /* int8 m x K row-major                       */
    const uint32_t *Xhat_dev; /* B x K field elements                       */
    uint32_t *Yhat_dev;       /* B x m field elements (output)              */
    int m, K, B;
} pvmvmd_mvm_batch_job;

/* The server's products for `count` independent batched requests, such as
 * the projections of one decoder layer for a batch of masked vectors
 * (Sec. 6.1: the server's online work is the product of each matrix with
 * the masked vectors it receives).  Results equal `count` calls of
 * pvmvmd_server_mvm.  Every job with B >= 2, K a multiple of 16 and a
 * 16-byte aligned W runs on the tensor cores in one persistent launch per
 * tile width (16-vector tiles for B <= 16, 64-vector tiles above; up to 8
 * jobs per launch): one pair of CTAs per pair of SMs walks a list of tiles
 * of all the jobs, longest first, so that small matrices fill the GPU and
 * the pipeline is set up once.  Other jobs take the path pvmvmd_server_mvm
 * gives them (batch-1 requests together in one grouped GEMV).  `jobs` is a host array that may be freed on return; outputs must
 * not overlap any input or each other.  1 <= count, each 1 <= K <=
 * PVMVMD_MAX_K, 1 <= m, 1 <= B.  The digit operands live in library scratch
 * held per stream, as for pvmvmd_server_mvm. */
int pvmvmd_server_mvm_grouped(const pvmvmd_mvm_batch_job *jobs, int count, void *stream);

/* Size of the fixed device buffer behind pvmvmd_server_mvm_noalloc. */
#define PVMVMD_NOALLOC_SCRATCH_BYTES (16u << 20)

/* The server's product Y_hat = M X_hat over F_q, like pvmvmd_server_mvm, but
 * without any memory allocation inside the call.  The paper has no
 * counterpart: this entry point exists for callers that cannot let the
 * library call cudaMalloc -- for instance a serving process whose device
 * memory is reserved up front by its own allocator or pool (a cudaMalloc
 * from inside the library could fail or fragment that pool), or a
 * latency-critical loop that cannot afford the regular call's first-use
 * allocation, or the device-wide synchronisation of replacing an outgrown
 * buffer.  It always runs the tensor-core digit product (also for B = 1),
 * whose fp16 digit tiles then live in one file-scope __device__ array of
 * PVMVMD_NOALLOC_SCRATCH_BYTES (16 MiB) that every GPU which loads the
 * library holds until the process exits.  The tiles take
 * ceil(B/64) * ceil(K/64) * 32 KiB, so for example B <= 64 allows
 * K <= 32768 and B <= 256 allows K <= 8192; a larger problem returns
 * PVMVMD_E_SHAPE and does nothing.  The first call on each device looks up
 * the array's device address (cudaGetSymbolAddress) with that device
 * current.  With CUDA's lazy module loading (the default) that lookup is
 * also when the device reserves the array, so make the first call on each
 * device before the caller reserves the rest of its device memory, and
 * before any stream capture; if the device cannot reserve the array then,
 * the call returns PVMVMD_E_NOMEM.  All calls share the one array, so calls
 * that overlap on the GPU (e.g. on two streams) race and give wrong
 * results; order them on one stream.  Arguments and results are those of
 * pvmvmd_server_mvm. */
int pvmvmd_server_mvm_noalloc(const int8_t *W_dev, int m, int K, const uint32_t *Xhat_dev, int B,
                              uint32_t *Yhat_dev, void *stream);

/* Verify and Decrypt (Protocol 3).  Verify: ell challenges e_q <- E_{t_y}^{N_y}
 * are drawn from challenge_key (repetition q reads nonce (10, 2q) and
 * (10, 2q+1)) and shared by all B vectors of the call, as Sec. 5.4 allows;
 * vector b is accepted iff (e_q^T Q) x_hat_b == e_q^T (G_y^T y_hat_b) for every q.
 * The right side is evaluated as (G_y e_q)^T y_hat_b, the same number by
 * transposition.  Decrypt: Y_b = y_hat_b - P e_x,b.  st_dev as written by
 * pvmvmd_encode (another state gives unspecified results, but every read
 * stays inside P); Xhat_dev B x K; Yhat_dev B x m; Y_dev B x m (may alias
 * Yhat_dev); accept_dev B int32, each 1 (accept) or 0 (reject).  A rejection
 * is data, not an error.  Y is written for rejected vectors too. */
int pvmvmd_decode_verify(pvmvmd_ctx *ctx, const void *st_dev, const uint32_t *Xhat_dev,
                         const uint32_t *Yhat_dev, int B, const pvmvmd_key *challenge_key,
                         uint32_t *Y_dev, int32_t *accept_dev, void *stream);

/* Boost mode (Sec. 7.2): the masks of a batch prepared ahead of the online
 * phase, while the client is idle, like preprocessed triples in MPC.
 *
 * pvmvmd_boost_prepare (offline) draws e_x for vectors numbered 0 .. B-1
 * under `key`, exactly as pvmvmd_encode would for the same key, and writes
 * the input masks Mask_in_b = G_x e_x,b (B x K), the output masks
 * Mask_out_b = P e_x,b (B x m) and st_b = e_x,b (pvmvmd_state_size bytes;
 * not needed online).  The online calls then cost one pass over the
 * vectors each:
 *   pvmvmd_boost_encode:  Xhat = X + Mask_in (B x K; Xhat may alias X or
 *                         Mask_in), the same Xhat pvmvmd_encode gives;
 *   pvmvmd_boost_decode_verify: as pvmvmd_decode_verify (fresh shared
 *                         challenges, same accept rule), with
 *                         Y = Yhat - Mask_out instead of the t_x rows of P.
 * A mask pair must be used for one vector only (Sec. 4.2 multi-query
 * privacy needs fresh masks per query). */
int pvmvmd_boost_prepare(pvmvmd_ctx *ctx, int B, const pvmvmd_key *key, uint32_t *mask_in_dev,
                         uint32_t *mask_out_dev, void *st_dev, void *stream);
int pvmvmd_boost_encode(const uint32_t *X_dev, const uint32_t *mask_in_dev, int B, int K,
                        uint32_t *Xhat_dev, void *stream);
int pvmvmd_boost_decode_verify(pvmvmd_ctx *ctx, const uint32_t *mask_out_dev,
                               const uint32_t *Xhat_dev, const uint32_t *Yhat_dev, int B,
                               const pvmvmd_key *challenge_key, uint32_t *Y_dev,
                               int32_t *accept_dev, void *stream);

/* ---------------------------------------------------------------------
 * Batch verification, Protocol 2 (Pi_Batch-vMVMD, Sec. 5): B claims
 * y_b = M_b x_b for B matrices of one shape m x n, checked together.  The
 * primary code G (dimension m, N = rate m) and the secondary code G'
 * (dimension B n, N' = rate B n) are sampled as code numbers 3 and 4 of
 * pvmvmd_code_sample_host.  Preprocess computes Q_b = G^T M_b, stored side
 * by side as Qs (N x B n, row i = (Q_1[i], ..., Q_B[i]) = Qt^T, the matrix
 * the server needs), and Qaux = Qt^T G' (stored transposed, N' x N).
 * A round:
 *   client pvmvmd_bv_challenge     once every y_b is fixed: ell primary
 *                                   challenges e^(q) <- E_t^N (tag 21),
 *                                   chal_dev ell x 2t (support, values);
 *   server pvmvmd_bv_server_project u^(q) = Qt e^(q), u_dev ell x B n;
 *   client pvmvmd_bv_check          draws ell' secondary challenges
 *                                   e'^(j) <- E_t'^N' (tag 22, key2) and
 *                                   sets *accept_dev (int32) to 1 iff
 *                                   e^(q)^T Qaux e'^(j) = (G' e'^(j))^T u^(q)
 *                                   for all q, j and
 *                                   u_b^(q)^T x_b = e^(q)^T G^T y_b for all
 *                                   b, q; else 0.
 * W_dev: B x m x n int8 (matrix b at W_dev + b m n); X_dev B x n; Y_dev
 * B x m.  Defaults (0 fields): rate 8, t = t' = 31, ell = ell' = 2. */
typedef struct pvmvmd_bv_ctx pvmvmd_bv_ctx;
typedef struct {
    int rate, t, ell, t2, ell2;
} pvmvmd_bv_params;
typedef struct {
    int B, m, n, rate, N, N2, t, ell, t2, ell2;
    const uint32_t *Qs, *QauxT, *chal2; /* device pointers owned by the context */
} pvmvmd_bv_view;
int pvmvmd_bv_preprocess(const int8_t *W_dev, int B, int m, int n, const pvmvmd_bv_params *params,
                         const pvmvmd_key *key, void *stream, pvmvmd_bv_ctx **out);
int pvmvmd_bv_challenge(pvmvmd_bv_ctx *ctx, const pvmvmd_key *key, uint32_t *chal_dev, void *stream);
int pvmvmd_bv_server_project(const pvmvmd_bv_ctx *ctx, const uint32_t *chal_dev, uint32_t *u_dev,
                             void *stream);
int pvmvmd_bv_check(pvmvmd_bv_ctx *ctx, const uint32_t *X_dev, const uint32_t *Y_dev,
                    const uint32_t *chal_dev, const uint32_t *u_dev, const pvmvmd_key *key2,
                    int32_t *accept_dev, void *stream);
int pvmvmd_bv_info(const pvmvmd_bv_ctx *ctx, pvmvmd_bv_view *view);
void pvmvmd_bv_destroy(pvmvmd_bv_ctx *ctx);

/* 16-bit weights.  Sec. 7.2 quantises FP8 weights as round(2^8 W), which can
 * exceed int8.  A 16-bit M (int16 m x K row-major, every entry in
 * [-32768, 32639]; others give unspecified results) is split once into two
 * int8 planes M = 256 M_hi + M_lo (M_lo the low byte read as signed), and
 * the server's product runs on both planes:
 *   pvmvmd_weights_split_i16   W -> Whi, Wlo (int8 m x K each);
 *   pvmvmd_server_mvm_i16      Yhat = Mhi Xhat * 256 + Mlo Xhat over F_q,
 *                              with Ytmp_dev (B x m) the caller's scratch;
 *   pvmvmd_preprocess_i16      as pvmvmd_preprocess for the 16-bit M
 *                              (encode, decode and verify then run
 *                              unchanged on the returned context). */
int pvmvmd_weights_split_i16(const int16_t *W_dev, int m, int K, int8_t *Whi_dev, int8_t *Wlo_dev,
                             void *stream);
int pvmvmd_server_mvm_i16(const int8_t *Whi_dev, const int8_t *Wlo_dev, int m, int K,
                          const uint32_t *Xhat_dev, int B, uint32_t *Yhat_dev, uint32_t *Ytmp_dev,
                          void *stream);
int pvmvmd_preprocess_i16(const int16_t *W_dev, int m, int K, const pvmvmd_params *params,
                          const pvmvmd_key *key, void *stream, pvmvmd_ctx **out);

/* The encoding Y = G^T X of one of a context's codes applied to L message
 * vectors held as lanes (App. B, encoding direction: G^T = A^T V2 Pi2^T A^T
 * V1 Pi1^T R^T, i.e. repeat r times, gather by pi1, scale by v1, prefix-sum,
 * gather by pi2, scale by v2, prefix-sum, all mod q).  This is the operation
 * pvmvmd_preprocess runs on the rows of M (P^T, which = 0) and its columns
 * (Q, which = 1).  which = 0 selects G_x (n = K), 1 selects G_y (n = m);
 * N = rate * n.  X_dev: n x L uint32 row-major (row i holds entry i of every
 * lane), canonical; Y_dev: N x L uint32 row-major.  scratch_dev: caller-owned
 * device memory of pvmvmd_code_encode_scratch bytes, 16-byte aligned, not
 * overlapping X_dev or Y_dev; its contents need no initialisation.  The call
 * allocates nothing and does not synchronise; it reads only the context's
 * code tables, so it may run beside any other call on the context.
 * Errors: PVMVMD_E_ARG for a null pointer or which outside {0, 1},
 * PVMVMD_E_SHAPE for L < 1; a look-back wait that expires is reported by
 * pvmvmd_device_status. */
int pvmvmd_code_encode_scratch(const pvmvmd_ctx *ctx, int which, int L, size_t *bytes);
int pvmvmd_code_encode_lanes(const pvmvmd_ctx *ctx, int which, const uint32_t *X_dev, int L,
                             uint32_t *Y_dev, void *scratch_dev, void *stream);

/* The number of kernels the library has enqueued in this process since it
 * was loaded, on every device and stream: each launch counts once when it is
 * enqueued, also while a stream is being captured.  Replaying a captured CUDA
 * graph launches its kernels again without passing through the library, so a
 * caller that replays a graph multiplies the count taken around the capture
 * by the replays.  (Introspection for benchmarks and tests; the paper has no
 * counterpart.) */
unsigned long long pvmvmd_kernel_launches(void);

/* Synchronise `stream`, then read and clear the library's device error word:
 * PVMVMD_E_DEVICE_TIMEOUT if any kernel gave up a bounded wait since the last
 * call, else PVMVMD_OK (or PVMVMD_E_CUDA if synchronisation failed). */
int pvmvmd_device_status(void *stream);

/* Test hook for the failure path of the bounded device waits (no paper
 * counterpart; off by default).  Every wait of the library's kernels on
 * another CTA or on the asynchronous units is bounded: when it expires the
 * kernel records PVMVMD_E_DEVICE_TIMEOUT in the device error word and
 * finishes (its results are then unspecified), instead of waiting forever.
 * This call lets a test make one such wait expire on purpose, with a short
 * limit, so that the expiry path itself runs:
 *   PVMVMD_DEBUG_WAIT_SCAN     the single-pass look-back scan of the syndrome
 *                              (encode of codes too long for a thread-block
 *                              cluster): tile `index` of every vector
 *                              publishes no status word, and look-back spins
 *                              give up after `limit` polls;
 *   PVMVMD_DEBUG_WAIT_PRODUCT  the tensor-core batched product: the second
 *                              CTA of every pair withholds its report for
 *                              K-block `index`, and pipeline waits give up
 *                              after `limit` nanoseconds;
 *   PVMVMD_DEBUG_WAIT_OFF      restore the normal behaviour (index and limit
 *                              ignored).
 * The setting is process-wide and is read when a kernel is launched (a
 * captured graph keeps the value it was captured with).  Returns
 * PVMVMD_E_ARG for an unknown site or a zero limit.  Not for production
 * use: every affected call gives wrong results. */
#define PVMVMD_DEBUG_WAIT_OFF 0
#define PVMVMD_DEBUG_WAIT_SCAN 1
#define PVMVMD_DEBUG_WAIT_PRODUCT 2
int pvmvmd_debug_expire_wait(int site, uint32_t index, uint64_t limit);

/* Fill *view with the context's public parameters. */
int pvmvmd_ctx_info(const pvmvmd_ctx *ctx, pvmvmd_ctx_view *view);

/* Release every device allocation of the context.  NULL is ignored. */
void pvmvmd_destroy(pvmvmd_ctx *ctx);

/* Static, human-readable text for a status code. */
const char *pvmvmd_strerror(int status);

/* Host-side sampling of one RAA generator exactly as pvmvmd_preprocess does
 * it (App. B): which = 0 for G_x, 1 for G_y; N = rate * dimension.  pi1/pi2
 * are Fisher-Yates permutations of [N] read from nonces (1+4*which, 0) and
 * (2+4*which, 0); v1/v2 are N uniform draws from F* read from nonces
 * (3+4*which, 0) and (4+4*which, 0).  Host arrays of length N.  Needs no GPU. */
int pvmvmd_code_sample_host(const pvmvmd_key *key, int which, uint32_t N, uint32_t *pi1,
                            uint32_t *pi2, uint32_t *v1, uint32_t *v2);

#ifdef __cplusplus
}
#endif

#endif /* PVMVMD_H */
