// C ABI of the pvMVMD library (include/pvmvmd.h): parameter resolution, the
// host-side sampling of the public RAA codes, context management, and the
// ordering of the device kernels for each protocol call.
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <atomic>
#include <mutex>
#include <new>
#include <vector>

#include "common.cuh"
#include "launch.h"

namespace pv {

// The library's device error word (kErr* bits).
__device__ uint32_t g_error_word = 0;

namespace {

// Domain tags of the ChaCha20 nonces (tag, index): the two codes, the masks
// and the challenges each read their own keystream.
constexpr uint32_t kTagCodeX = 1;       // G_x: pi1 = 1, pi2 = 2, v1 = 3, v2 = 4
constexpr uint32_t kTagCodeY = 5;       // G_y: pi1 = 5, pi2 = 6, v1 = 7, v2 = 8
static_assert(kTagCodeY == kTagCodeX + 4, "code `which` reads tags kTagCodeX + 4 which + 0..3");
constexpr uint32_t kTagMask = 9;
constexpr uint32_t kTagChallenge = 10;
constexpr uint32_t kTagBvPrimary = 21;    // batch verification challenges
constexpr uint32_t kTagBvSecondary = 22;
// Encode batches of at least this many vectors as the lanes of N x B arrays
// (launch_lane_syndrome) when the code needs a cluster per vector; smaller
// batches and codes that fit one CTA use the fused kernel.
constexpr int kLaneMinBatch = 32;
// Server products of at most this many vectors use the small-batch GEMV.
constexpr int kSmallBatchMax = 16;

// --------------------------------------------------------------------------
// Host ChaCha20 keystream (RFC 8439 Sec. 2.3) read as 32-bit words.
// --------------------------------------------------------------------------
class KeyStream {
  public:
    KeyStream(const pvmvmd_key &key, uint32_t tag, uint64_t index) : key_(key) {
        nonce_[0] = tag;
        nonce_[1] = (uint32_t)index;
        nonce_[2] = (uint32_t)(index >> 32);
    }
    uint32_t word() {
        if (used_ == 16) refill();
        return block_[used_++];
    }
    // Uniform in [0, k): top bitlen(k-1) bits, rejected while >= k.
    uint32_t below(uint32_t k) {
        if (k <= 1) return 0;
        int bits = 0;
        for (uint32_t v = k - 1; v; v >>= 1) ++bits;
        for (;;) {
            const uint32_t v = word() >> (32 - bits);
            if (v < k) return v;
        }
    }
    // Uniform in F* = [1, q): top 31 bits, rejected outside [1, q).
    uint32_t nonzero_field() {
        for (;;) {
            const uint32_t v = word() >> 1;
            if (v != 0 && v < kQ) return v;
        }
    }

  private:
    static uint32_t rotl(uint32_t v, int c) { return (v << c) | (v >> (32 - c)); }
    static void quarter(uint32_t *s, int a, int b, int c, int d) {
        s[a] += s[b]; s[d] = rotl(s[d] ^ s[a], 16);
        s[c] += s[d]; s[b] = rotl(s[b] ^ s[c], 12);
        s[a] += s[b]; s[d] = rotl(s[d] ^ s[a], 8);
        s[c] += s[d]; s[b] = rotl(s[b] ^ s[c], 7);
    }
    void refill() {
        uint32_t in[16] = {0x61707865u, 0x3320646eu, 0x79622d32u, 0x6b206574u};
        std::memcpy(in + 4, key_.k, sizeof key_.k);
        in[12] = counter_++;
        in[13] = nonce_[0];
        in[14] = nonce_[1];
        in[15] = nonce_[2];
        uint32_t s[16];
        std::memcpy(s, in, sizeof s);
        for (int i = 0; i < 10; ++i) {
            quarter(s, 0, 4, 8, 12); quarter(s, 1, 5, 9, 13);
            quarter(s, 2, 6, 10, 14); quarter(s, 3, 7, 11, 15);
            quarter(s, 0, 5, 10, 15); quarter(s, 1, 6, 11, 12);
            quarter(s, 2, 7, 8, 13); quarter(s, 3, 4, 9, 14);
        }
        for (int i = 0; i < 16; ++i) block_[i] = s[i] + in[i];
        used_ = 0;
    }
    pvmvmd_key key_;
    uint32_t nonce_[3];
    uint32_t counter_ = 0;
    uint32_t block_[16];
    int used_ = 16;
};

void sample_code_host(const pvmvmd_key &key, int which, uint32_t N, uint32_t *pi1, uint32_t *pi2,
                      uint32_t *v1, uint32_t *v2) {
    // code `which` reads tags 4 which + 1 .. 4 which + 4 (G_x = 0, G_y = 1;
    // the batch verification codes are 3 and 4)
    const uint32_t tag0 = kTagCodeX + 4u * (uint32_t)which;
    uint32_t *perms[2] = {pi1, pi2};
    for (int p = 0; p < 2; ++p) {  // Fisher-Yates, last index first
        KeyStream ks(key, tag0 + p, 0);
        uint32_t *a = perms[p];
        for (uint32_t i = 0; i < N; ++i) a[i] = i;
        for (uint32_t i = N; i-- > 1;) {
            const uint32_t j = ks.below(i + 1);
            const uint32_t tmp = a[i];
            a[i] = a[j];
            a[j] = tmp;
        }
    }
    uint32_t *scales[2] = {v1, v2};
    for (int p = 0; p < 2; ++p) {
        KeyStream ks(key, tag0 + 2 + p, 0);
        for (uint32_t i = 0; i < N; ++i) scales[p][i] = ks.nonzero_field();
    }
}

// --------------------------------------------------------------------------
// Device helpers
// --------------------------------------------------------------------------
int check_device() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PVMVMD_E_NODEVICE;
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
        return PVMVMD_E_NODEVICE;
    return (major == 10 && minor == 3) ? PVMVMD_OK : PVMVMD_E_NODEVICE;
}

std::atomic<unsigned long long> g_kernel_launches{0};
unsigned long long kernel_launches() { return g_kernel_launches.load(std::memory_order_relaxed); }
}  // namespace
void note_launch() { g_kernel_launches.fetch_add(1, std::memory_order_relaxed); }
namespace {
uint32_t *error_word() {
    static std::mutex mu;
    static uint32_t *addr[64] = {nullptr};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) return nullptr;
        addr[dev] = static_cast<uint32_t *>(p);
    }
    return addr[dev];
}

#define PV_CUDA(expr)                                  \
    do {                                               \
        cudaError_t e_ = (expr);                       \
        if (e_ != cudaSuccess) {                       \
            (void)cudaGetLastError();                  \
            return e_ == cudaErrorMemoryAllocation ? PVMVMD_E_NOMEM : PVMVMD_E_CUDA; \
        }                                              \
    } while (0)

template <typename T>
cudaError_t dev_alloc(T **p, size_t count) {
    *p = nullptr;
    if (count == 0) count = 1;
    return cudaMalloc(reinterpret_cast<void **>(p), count * sizeof(T));
}

struct CodeDev {
    uint32_t *pi1 = nullptr, *pi2 = nullptr, *v1 = nullptr, *v2 = nullptr;
    uint32_t *pi1inv = nullptr, *pi2inv = nullptr, *v2p = nullptr;
    uint32_t *v2m = nullptr, *v1pm = nullptr;  // Montgomery-scaled v2 and v1 o pi1^-1
    uint32_t *v1m = nullptr;                   // Montgomery-scaled v1
};

}  // namespace
}  // namespace pv

struct pvmvmd_ctx {
    int device = 0;
    pvmvmd_params params{};
    int m = 0, K = 0, rate = 0, Nx = 0, Ny = 0, t_x = 0, t_y = 0, ell = 0, sb = 0;
    pv::CodeDev gx, gy;
    uint32_t *PT = nullptr, *Q = nullptr;
    uint32_t *F = nullptr, *Fy = nullptr, *chal = nullptr, *g = nullptr, *u = nullptr;
    // scan status words of the encode (status) and of the challenges
    // (status_y): an encode and a decode share no scratch
    unsigned long long *status = nullptr, *status_y = nullptr;
    // lane-parallel encode scratch (null when scratch_batch < kLaneMinBatch)
    uint32_t *S = nullptr, *laux = nullptr;
    // decode: the challenge kernels run on `side` (highest stream priority),
    // forked from and joined back to the caller's stream, while the decrypt
    // streams P^T
    cudaStream_t side = nullptr;
    cudaEvent_t fork = nullptr, join = nullptr;
    std::vector<void *> owned;
};

// Batch verification (Protocol 2) for B matrices of one shape m x n.
struct pvmvmd_bv_ctx {
    int device = 0;
    int B = 0, m = 0, n = 0, rate = 0, N = 0, N2 = 0, t = 0, ell = 0, t2 = 0, ell2 = 0;
    pv::CodeDev g, g2;       // primary code (dimension m), secondary code (dimension B n)
    uint32_t *Qs = nullptr;    // N x B n: row i = (Q_1[i], ..., Q_B[i]) = Qt^T (public)
    uint32_t *QauxT = nullptr; // N' x N: Qaux transposed
    uint32_t *Yt = nullptr, *Z = nullptr;  // m x B, N x B
    uint32_t *chal2 = nullptr, *R = nullptr, *F2 = nullptr;
    uint32_t *eS = nullptr, *eticket = nullptr;  // encode scratch: S, scan ticket
    unsigned long long *estatus = nullptr;       // and scan status words
    unsigned long long *status = nullptr;
    std::vector<void *> owned;
};

namespace pv {
namespace {

template <typename Ctx, typename T>
cudaError_t ctx_alloc(Ctx *c, T **p, size_t count) {
    cudaError_t e = dev_alloc(p, count);
    if (e == cudaSuccess) c->owned.push_back(*p);
    return e;
}

template <typename Ctx>
int upload_code(Ctx *c, CodeDev &d, const pvmvmd_key &key, int which, uint32_t N, cudaStream_t s) {
    std::vector<uint32_t> pi1(N), pi2(N), v1(N), v2(N), pi1inv(N), pi2inv(N), v2p(N), v2m(N), v1pm(N), v1m(N);
    sample_code_host(key, which, N, pi1.data(), pi2.data(), v1.data(), v2.data());
    for (uint32_t j = 0; j < N; ++j) {
        pi1inv[pi1[j]] = j;
        pi2inv[pi2[j]] = j;
    }
    for (uint32_t i = 0; i < N; ++i) {
        v2p[i] = v2[pi2inv[i]];
        v2m[i] = to_mont(v2[i]);
        v1pm[i] = to_mont(v1[pi1inv[i]]);
        v1m[i] = to_mont(v1[i]);
    }
    uint32_t **dst[10] = {&d.pi1, &d.pi2, &d.v1, &d.v2, &d.pi1inv, &d.pi2inv, &d.v2p, &d.v2m, &d.v1pm, &d.v1m};
    const std::vector<uint32_t> *src[10] = {&pi1, &pi2, &v1, &v2, &pi1inv, &pi2inv, &v2p, &v2m, &v1pm, &v1m};
    for (int i = 0; i < 10; ++i) {
        PV_CUDA(ctx_alloc(c, dst[i], N));
        PV_CUDA(cudaMemcpyAsync(*dst[i], src[i]->data(), (size_t)N * 4, cudaMemcpyHostToDevice, s));
    }
    // the host vectors are released on return; wait for the copies
    PV_CUDA(cudaStreamSynchronize(s));
    return PVMVMD_OK;
}

// Y (N x L lanes, row stride ldy) = G^T applied to the L lanes of X (n x L,
// row stride ldx; row i holds message entry i of every lane), in lane chunks.
// One chunk of lanes with caller-provided scratch (S: N x nl; status:
// encode_scan_status_words(N, nl) 64-bit words; ticket: one word); no
// allocation, no sync.
int encode_lanes_into(const CodeDev &d, uint32_t n, uint32_t r, const void *X, bool x_is_i8, size_t ldx,
                      uint32_t nl, uint32_t *Y, size_t ldy, uint32_t *S, unsigned long long *status,
                      uint32_t *ticket, uint32_t *err, cudaStream_t s) {
    const uint32_t N = n * r;
    cudaError_t e = encode_scan_clear(status, ticket, N, nl, s);
    if (e == cudaSuccess)  // S = A^T V1 Pi1^T R^T X
        e = launch_encode_scan(X, x_is_i8, ldx, d.pi1, r, d.v1m, N, nl, S, nl, status, ticket, err, s);
    if (e == cudaSuccess) e = encode_scan_clear(status, ticket, N, nl, s);
    if (e == cudaSuccess)  // Y = A^T V2 Pi2^T S
        e = launch_encode_scan(S, false, nl, d.pi2, 1, d.v2m, N, nl, Y, ldy, status, ticket, err, s);
    return e == cudaSuccess ? PVMVMD_OK : PVMVMD_E_CUDA;
}

// Y (N x L lanes, row stride ldy) = G^T applied to the L lanes of X (n x L,
// row stride ldx; row i holds message entry i of every lane; int8 or
// uint32), in lane chunks with scratch allocated here (preprocessing only).
int encode_lanes(const CodeDev &d, uint32_t n, uint32_t r, const void *X, bool x_is_i8, size_t ldx,
                 uint32_t L, uint32_t *Y, size_t ldy, uint32_t *err, cudaStream_t s) {
    const uint32_t N = n * r;
    size_t lc = ((size_t)1 << 28) / N;  // lanes per chunk: about 1 GiB of scratch
    lc = (lc / 256) * 256;
    if (lc < 256) lc = 256;
    if (lc > L) lc = L;
    uint32_t *S = nullptr, *ticket = nullptr;
    unsigned long long *status = nullptr;
    const size_t sw = encode_scan_status_words(N, (uint32_t)lc);
    int status_code = PVMVMD_OK;
    if (dev_alloc(&S, (size_t)N * lc) != cudaSuccess || dev_alloc(&status, sw) != cudaSuccess ||
        dev_alloc(&ticket, 1) != cudaSuccess) {
        status_code = PVMVMD_E_NOMEM;
    }
    for (uint32_t l0 = 0; status_code == PVMVMD_OK && l0 < L; l0 += (uint32_t)lc) {
        const uint32_t nl = (uint32_t)((L - l0) < lc ? (L - l0) : lc);
        const void *Xl = x_is_i8 ? static_cast<const void *>(static_cast<const int8_t *>(X) + l0)
                                 : static_cast<const void *>(static_cast<const uint32_t *>(X) + l0);
        status_code = encode_lanes_into(d, n, r, Xl, x_is_i8, ldx, nl, Y + l0, ldy, S, status, ticket, err, s);
    }
    if (cudaStreamSynchronize(s) != cudaSuccess) status_code = PVMVMD_E_CUDA;
    cudaFree(S);
    cudaFree(status);
    cudaFree(ticket);
    return status_code;
}

int read_and_clear_error() {
    uint32_t *ew = error_word();
    if (!ew) return PVMVMD_E_CUDA;
    uint32_t v = 0;
    if (cudaMemcpy(&v, ew, 4, cudaMemcpyDeviceToHost) != cudaSuccess) return PVMVMD_E_CUDA;
    if (v) {
        const uint32_t zero = 0;
        if (cudaMemcpy(ew, &zero, 4, cudaMemcpyHostToDevice) != cudaSuccess) return PVMVMD_E_CUDA;
        return PVMVMD_E_DEVICE_TIMEOUT;
    }
    return PVMVMD_OK;
}

}  // namespace

uint32_t *library_error_word() { return error_word(); }

namespace {
std::mutex g_debug_mu;
DebugWait g_debug;
}  // namespace

DebugWait debug_wait() {
    std::lock_guard<std::mutex> lock(g_debug_mu);
    return g_debug;
}

}  // namespace pv

using namespace pv;

extern "C" {

const char *pvmvmd_strerror(int status) {
    switch (status) {
        case PVMVMD_OK: return "success";
        case PVMVMD_E_ARG: return "invalid argument (null pointer or bad value)";
        case PVMVMD_E_SHAPE: return "shape or batch size outside the supported range";
        case PVMVMD_E_PARAM: return "inconsistent protocol parameters (e.g. t > N)";
        case PVMVMD_E_CUDA: return "a CUDA runtime call or kernel launch failed";
        case PVMVMD_E_NOMEM: return "out of memory";
        case PVMVMD_E_DEVICE_TIMEOUT: return "a bounded device-side wait expired";
        case PVMVMD_E_NODEVICE: return "no sm_103 (GB300) CUDA device is current";
        default: return "unknown status";
    }
}

int pvmvmd_params_resolve(const pvmvmd_params *in, int m, int K, pvmvmd_params *out) {
    if (!out || m < 1 || K < 1) return PVMVMD_E_ARG;
    pvmvmd_params p{};
    if (in) p = *in;
    if (p.lambda < 0 || p.kappa < 0 || p.rate < 0 || p.delta < 0 || p.t_x < 0 || p.t_y < 0 ||
        p.ell < 0 || p.scratch_batch < 0 || p.delta >= 1.0)
        return PVMVMD_E_PARAM;
    if (p.lambda == 0) p.lambda = 128;
    if (p.kappa == 0) p.kappa = 40;
    if (p.rate == 0) p.rate = 8;
    if (p.delta == 0) p.delta = 0.5;
    if (p.scratch_batch == 0) p.scratch_batch = 64;
    const double Nx = (double)p.rate * K, Ny = (double)p.rate * m;
    if (Nx > 4294967295.0 || Ny > 4294967295.0) return PVMVMD_E_SHAPE;
    if (p.t_x == 0) {  // Eq. (1)
        const double t = std::ceil(std::log(2.0) * ((double)p.lambda - std::log2(Nx)) / p.delta);
        p.t_x = t < 1 ? 1 : (int)t;
    }
    // Thm 5.2, by the two cases of its proof: with lf = log2(|F| - 1),
    // case 1 (lf >= kappa + 1) needs (1-delta)^t <= 2^-(kappa+1) and ell = 1;
    // case 2 needs (1-delta)^t <= 1/(|F|-1) and ell = ceil(kappa / (lf - 1)).
    const double lf = std::log2((double)(kQ - 1));
    const double per = -std::log2(1.0 - p.delta);
    const bool case1 = lf >= p.kappa + 1;
    if (p.t_y == 0) p.t_y = (int)std::ceil((case1 ? (double)(p.kappa + 1) : lf) / per);
    if (p.ell == 0) p.ell = case1 ? 1 : (int)std::ceil((double)p.kappa / (lf - 1.0));
    if (p.t_x > Nx || p.t_y > Ny || p.t_x > PVMVMD_MAX_T || p.t_y > PVMVMD_MAX_T || p.ell > 16 ||
        p.ell < 1)
        return PVMVMD_E_PARAM;
    *out = p;
    return PVMVMD_OK;
}

int pvmvmd_code_sample_host(const pvmvmd_key *key, int which, uint32_t N, uint32_t *pi1,
                            uint32_t *pi2, uint32_t *v1, uint32_t *v2) {
    if (!key || !pi1 || !pi2 || !v1 || !v2 || (which != 0 && which != 1)) return PVMVMD_E_ARG;
    sample_code_host(*key, which, N, pi1, pi2, v1, v2);
    return PVMVMD_OK;
}

void pvmvmd_destroy(pvmvmd_ctx *ctx) {
    if (!ctx) return;
    int cur = 0;
    cudaGetDevice(&cur);
    cudaSetDevice(ctx->device);
    for (void *p : ctx->owned) cudaFree(p);
    if (ctx->fork) cudaEventDestroy(ctx->fork);
    if (ctx->join) cudaEventDestroy(ctx->join);
    if (ctx->side) cudaStreamDestroy(ctx->side);
    cudaSetDevice(cur);
    delete ctx;
}

namespace pv {
namespace {
int preprocess_impl(const void *W_dev, bool w16, int m, int K, const pvmvmd_params *params,
                    const pvmvmd_key *key, void *stream, pvmvmd_ctx **out);
}  // namespace
}  // namespace pv

int pvmvmd_preprocess(const int8_t *W_dev, int m, int K, const pvmvmd_params *params,
                      const pvmvmd_key *key, void *stream, pvmvmd_ctx **out) {
    return pv::preprocess_impl(W_dev, false, m, K, params, key, stream, out);
}

int pvmvmd_preprocess_i16(const int16_t *W_dev, int m, int K, const pvmvmd_params *params,
                          const pvmvmd_key *key, void *stream, pvmvmd_ctx **out) {
    return pv::preprocess_impl(W_dev, true, m, K, params, key, stream, out);
}

namespace pv {
namespace {
int preprocess_impl(const void *W_dev, bool w16, int m, int K, const pvmvmd_params *params,
                    const pvmvmd_key *key, void *stream, pvmvmd_ctx **out) {
    if (!out) return PVMVMD_E_ARG;
    *out = nullptr;
    if (!W_dev || !key) return PVMVMD_E_ARG;
    if (m < 1 || K < 1 || K > PVMVMD_MAX_K) return PVMVMD_E_SHAPE;
    int st = check_device();
    if (st) return st;
    pvmvmd_params p;
    st = pvmvmd_params_resolve(params, m, K, &p);
    if (st) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;

    pvmvmd_ctx *c = new (std::nothrow) pvmvmd_ctx();
    if (!c) return PVMVMD_E_NOMEM;
    cudaGetDevice(&c->device);
    c->params = p;
    c->m = m;
    c->K = K;
    c->rate = p.rate;
    c->Nx = p.rate * K;
    c->Ny = p.rate * m;
    c->t_x = p.t_x;
    c->t_y = p.t_y;
    c->ell = p.ell;
    c->sb = p.scratch_batch;

    auto fail = [&](int code) {
        pvmvmd_destroy(c);
        return code;
    };
    if ((st = upload_code(c, c->gx, *key, 0, c->Nx, s))) return fail(st);
    if ((st = upload_code(c, c->gy, *key, 1, c->Ny, s))) return fail(st);
    if (ctx_alloc(c, &c->PT, (size_t)c->Nx * m) != cudaSuccess ||
        ctx_alloc(c, &c->Q, (size_t)c->Ny * K) != cudaSuccess ||
        ctx_alloc(c, &c->F, (size_t)((c->sb + 3) & ~3) * c->Nx) != cudaSuccess ||  // lanes padded to 4
        ctx_alloc(c, &c->Fy, (size_t)c->ell * c->Ny) != cudaSuccess ||
        ctx_alloc(c, &c->chal, (size_t)c->ell * 2 * c->t_y) != cudaSuccess ||
        ctx_alloc(c, &c->g, (size_t)c->ell * m) != cudaSuccess ||
        ctx_alloc(c, &c->u, (size_t)c->ell * K) != cudaSuccess ||
        ctx_alloc(c, &c->status, scan_status_words(c->Nx, c->sb)) != cudaSuccess ||
        ctx_alloc(c, &c->status_y, scan_status_words(c->Ny, c->ell)) != cudaSuccess)
        return fail(PVMVMD_E_NOMEM);
    // the challenge kernels are few and short; at the highest priority their
    // blocks take SMs as the decrypt's blocks drain instead of queueing
    // behind the rest of the decrypt's grid
    int prio_least = 0, prio_greatest = 0;
    if (cudaDeviceGetStreamPriorityRange(&prio_least, &prio_greatest) != cudaSuccess ||
        cudaStreamCreateWithPriority(&c->side, cudaStreamNonBlocking, prio_greatest) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->fork, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->join, cudaEventDisableTiming) != cudaSuccess)
        return fail(PVMVMD_E_CUDA);
    if (c->sb >= kLaneMinBatch &&
        (ctx_alloc(c, &c->S, lane_state_words(c->t_x, c->sb)) != cudaSuccess ||
         ctx_alloc(c, &c->laux, lane_aux_words(c->Nx, c->sb)) != cudaSuccess))
        return fail(PVMVMD_E_NOMEM);

    if (w16) {
        // 16-bit M: lift it to F_q, then encode as uint32 lanes
        uint32_t *M32 = nullptr, *MT32 = nullptr;
        if (dev_alloc(&M32, (size_t)m * K) != cudaSuccess || dev_alloc(&MT32, (size_t)m * K) != cudaSuccess) {
            cudaFree(M32);
            return fail(PVMVMD_E_NOMEM);
        }
        if (launch_lift_i16(static_cast<const int16_t *>(W_dev), (size_t)m * K, M32, s) != cudaSuccess ||
            launch_transpose_u32(M32, m, K, MT32, s) != cudaSuccess) {
            cudaFree(M32);
            cudaFree(MT32);
            return fail(PVMVMD_E_CUDA);
        }
        st = encode_lanes(c->gx, K, c->rate, MT32, false, (size_t)m, m, c->PT, (size_t)m, err, s);
        if (!st) st = encode_lanes(c->gy, m, c->rate, M32, false, (size_t)K, K, c->Q, (size_t)K, err, s);
        cudaFree(M32);
        cudaFree(MT32);
        if (st) return fail(st);
        if ((st = read_and_clear_error())) return fail(st);
        *out = c;
        return PVMVMD_OK;
    }
    // P^T = G_x^T M^T: the m rows of M are the lanes, so transpose M first.
    int8_t *MT = nullptr;
    if (dev_alloc(&MT, (size_t)m * K) != cudaSuccess) return fail(PVMVMD_E_NOMEM);
    if (launch_transpose_i8(static_cast<const int8_t *>(W_dev), m, K, MT, s) != cudaSuccess) {
        cudaFree(MT);
        return fail(PVMVMD_E_CUDA);
    }
    st = encode_lanes(c->gx, K, c->rate, MT, true, (size_t)m, m, c->PT, (size_t)m, err, s);
    cudaFree(MT);
    if (st) return fail(st);
    // Q = G_y^T M: the K columns of M are the lanes.
    st = encode_lanes(c->gy, m, c->rate, W_dev, true, (size_t)K, K, c->Q, (size_t)K, err, s);
    if (st) return fail(st);
    if ((st = read_and_clear_error())) return fail(st);
    *out = c;
    return PVMVMD_OK;
}
}  // namespace
}  // namespace pv

int pvmvmd_weights_split_i16(const int16_t *W_dev, int m, int K, int8_t *Whi_dev, int8_t *Wlo_dev,
                             void *stream) {
    using namespace pv;
    if (!W_dev || !Whi_dev || !Wlo_dev) return PVMVMD_E_ARG;
    if (m < 1 || K < 1) return PVMVMD_E_SHAPE;
    PV_CUDA(launch_split_i16(W_dev, (size_t)m * K, Whi_dev, Wlo_dev, static_cast<cudaStream_t>(stream)));
    return PVMVMD_OK;
}

int pvmvmd_server_mvm_i16(const int8_t *Whi_dev, const int8_t *Wlo_dev, int m, int K, const uint32_t *Xhat_dev,
                          int B, uint32_t *Yhat_dev, uint32_t *Ytmp_dev, void *stream) {
    using namespace pv;
    if (!Whi_dev || !Wlo_dev || !Ytmp_dev) return PVMVMD_E_ARG;
    int st = pvmvmd_server_mvm(Whi_dev, m, K, Xhat_dev, B, Yhat_dev, stream);
    if (st) return st;
    st = pvmvmd_server_mvm(Wlo_dev, m, K, Xhat_dev, B, Ytmp_dev, stream);
    if (st) return st;
    PV_CUDA(launch_combine_256(Yhat_dev, Ytmp_dev, (size_t)B * m, static_cast<cudaStream_t>(stream)));
    return PVMVMD_OK;
}

int pvmvmd_state_size(const pvmvmd_ctx *ctx, int B, size_t *bytes) {
    if (!ctx || !bytes || B < 0) return PVMVMD_E_ARG;
    *bytes = (size_t)B * 2 * ctx->t_x * sizeof(uint32_t);
    return PVMVMD_OK;
}

namespace pv {
namespace {
// Xhat = X + G_x e_x for the B vectors (X null: Xhat = G_x e_x alone).
int encode_batch(pvmvmd_ctx *ctx, const uint32_t *X_dev, int B, const pvmvmd_key *key,
                 uint32_t *Xhat_dev, void *st_dev, cudaStream_t s);
}  // namespace
}  // namespace pv

int pvmvmd_encode(pvmvmd_ctx *ctx, const uint32_t *X_dev, int B, const pvmvmd_key *key,
                  uint32_t *Xhat_dev, void *st_dev, void *stream) {
    if (!ctx || !X_dev || !key || !Xhat_dev || !st_dev) return PVMVMD_E_ARG;
    if (B < 1) return PVMVMD_E_SHAPE;
    return pv::encode_batch(ctx, X_dev, B, key, Xhat_dev, st_dev, static_cast<cudaStream_t>(stream));
}

int pvmvmd_boost_prepare(pvmvmd_ctx *ctx, int B, const pvmvmd_key *key, uint32_t *mask_in_dev,
                         uint32_t *mask_out_dev, void *st_dev, void *stream) {
    using namespace pv;
    if (!ctx || !key || !mask_in_dev || !mask_out_dev || !st_dev) return PVMVMD_E_ARG;
    if (B < 1) return PVMVMD_E_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int st = encode_batch(ctx, nullptr, B, key, mask_in_dev, st_dev, s);
    if (st != PVMVMD_OK) return st;
    PV_CUDA(launch_output_mask(ctx->PT, ctx->m, static_cast<const uint32_t *>(st_dev), ctx->t_x, B,
                               mask_out_dev, s));
    return PVMVMD_OK;
}

int pvmvmd_boost_encode(const uint32_t *X_dev, const uint32_t *mask_in_dev, int B, int K,
                        uint32_t *Xhat_dev, void *stream) {
    using namespace pv;
    if (!X_dev || !mask_in_dev || !Xhat_dev) return PVMVMD_E_ARG;
    if (B < 1 || K < 1) return PVMVMD_E_SHAPE;
    PV_CUDA(launch_field_add(X_dev, mask_in_dev, (size_t)B * K, Xhat_dev,
                             static_cast<cudaStream_t>(stream)));
    return PVMVMD_OK;
}

namespace pv {
namespace {
int encode_batch(pvmvmd_ctx *ctx, const uint32_t *X_dev, int B, const pvmvmd_key *key,
                 uint32_t *Xhat_dev, void *st_dev, cudaStream_t s) {
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;
    uint32_t *stp = static_cast<uint32_t *>(st_dev);
    const CodeDev &d = ctx->gx;
    int C;
    uint32_t slice;
    size_t smem;
    const bool fused = syndrome_fused_plan(ctx->Nx, ctx->t_x, &C, &slice, &smem);
    if (B >= kLaneMinBatch && ctx->laux && !(fused && C == 1)) {
        // vectors as lanes: every permutation step moves whole rows (a code
        // that fits one CTA's shared memory stays on chip in the fused kernel)
        for (int b0 = 0; b0 < B; b0 += ctx->sb) {
            const uint32_t L = (uint32_t)(B - b0 < ctx->sb ? B - b0 : ctx->sb);
            PV_CUDA(launch_lane_syndrome(*key, kTagMask, (uint64_t)b0, ctx->Nx, ctx->t_x, L, d.pi2,
                                         d.v2m, d.v1m, d.pi1inv, ctx->K, ctx->rate,
                                         stp + (size_t)b0 * 2 * ctx->t_x, ctx->S, ctx->F, ctx->laux,
                                         X_dev ? X_dev + (size_t)b0 * ctx->K : nullptr,
                                         Xhat_dev + (size_t)b0 * ctx->K, s));
        }
        return PVMVMD_OK;
    }
    if (fused) {
        // sample, scan and gather in one launch per batch, no scratch
        PV_CUDA(launch_syndrome_fused(*key, kTagMask, 0, ctx->Nx, ctx->t_x, (uint32_t)B, d.pi2inv,
                                      d.v2p, d.v1, d.pi1inv, d.pi2, d.v2m, d.v1pm, ctx->K, ctx->rate,
                                      stp, X_dev, Xhat_dev, s, /*pdl=*/true, kSpreadEncode));
        return PVMVMD_OK;
    }
    for (int b0 = 0; b0 < B; b0 += ctx->sb) {
        const uint32_t nb = (uint32_t)(B - b0 < ctx->sb ? B - b0 : ctx->sb);
        uint32_t *e = stp + (size_t)b0 * 2 * ctx->t_x;
        PV_CUDA(launch_sample_sparse(*key, kTagMask, (uint64_t)b0, ctx->Nx, ctx->t_x, nb, e,
                                     ctx->status, scan_status_words(ctx->Nx, nb), s));
        PV_CUDA(launch_syndrome_scan(d.pi2inv, d.v2p, d.v1, ctx->Nx, e, ctx->t_x, nb, ctx->F,
                                     ctx->status, err, s));
        PV_CUDA(launch_syndrome_gather(d.pi1inv, ctx->K, ctx->rate, ctx->F, ctx->Nx,
                                       X_dev ? X_dev + (size_t)b0 * ctx->K : nullptr,
                                       Xhat_dev + (size_t)b0 * ctx->K, nb, s));
    }
    return PVMVMD_OK;
}
}  // namespace
}  // namespace pv

int pvmvmd_server_mvm(const int8_t *W_dev, int m, int K, const uint32_t *Xhat_dev, int B,
                      uint32_t *Yhat_dev, void *stream) {
    if (!W_dev || !Xhat_dev || !Yhat_dev) return PVMVMD_E_ARG;
    if (m < 1 || K < 1 || K > PVMVMD_MAX_K || B < 1) return PVMVMD_E_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;
    if (B == 1) {
        PV_CUDA(launch_gemv(W_dev, m, K, Xhat_dev, Yhat_dev, err, s));
        return PVMVMD_OK;
    }
    // a few vectors: one pass over M per four vectors with dp4a, unless the
    // problem is large enough for the tensor-core product with 16-vector
    // tiles to win (measured: 14336 x 4096 with 8 vectors 41.0 against
    // 27.1 us, with 4 vectors 23.8 against 26.0 us; 4096 x 2560 with 8
    // vectors 12.1 against 12.9 us)
    const bool tensor_small = B >= 8 && (double)m * K * B >= 128.0 * 1024 * 1024;
    if (B <= kSmallBatchMax && !tensor_small && K % 16 == 0 &&
        ((reinterpret_cast<uintptr_t>(W_dev) | reinterpret_cast<uintptr_t>(Xhat_dev)) & 15u) == 0) {
        PV_CUDA(launch_gemv_small_batch(W_dev, m, K, Xhat_dev, B, Yhat_dev, s));
        return PVMVMD_OK;
    }
    PV_CUDA(launch_batched(W_dev, m, K, Xhat_dev, B, Yhat_dev, err, s));
    return PVMVMD_OK;
}

int pvmvmd_server_mvm_multi(const pvmvmd_mvm_job *jobs, int count, void *stream) {
    if (!jobs || count < 1) return count < 1 ? PVMVMD_E_SHAPE : PVMVMD_E_ARG;
    for (int i = 0; i < count; ++i) {
        const pvmvmd_mvm_job &j = jobs[i];
        if (!j.W_dev || !j.xhat_dev || !j.yhat_dev) return PVMVMD_E_ARG;
        if (j.m < 1 || j.K < 1 || j.K > PVMVMD_MAX_K) return PVMVMD_E_SHAPE;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;
    std::vector<MvmJob> grouped;
    grouped.reserve(count);
    for (int i = 0; i < count; ++i) {
        const pvmvmd_mvm_job &j = jobs[i];
        MvmJob t{j.W_dev, j.xhat_dev, j.yhat_dev, j.m, j.K, (size_t)j.K, 0};
        if (multi_eligible(t))
            grouped.push_back(t);
        else
            PV_CUDA(launch_gemv(j.W_dev, j.m, j.K, j.xhat_dev, j.yhat_dev, err, s));
    }
    if (!grouped.empty()) PV_CUDA(launch_gemv_multi(grouped.data(), (int)grouped.size(), s));
    return PVMVMD_OK;
}

int pvmvmd_server_mvm_grouped(const pvmvmd_mvm_batch_job *jobs, int count, void *stream) {
    if (!jobs || count < 1) return count < 1 ? PVMVMD_E_SHAPE : PVMVMD_E_ARG;
    for (int i = 0; i < count; ++i) {
        const pvmvmd_mvm_batch_job &j = jobs[i];
        if (!j.W_dev || !j.Xhat_dev || !j.Yhat_dev) return PVMVMD_E_ARG;
        if (j.m < 1 || j.K < 1 || j.K > PVMVMD_MAX_K || j.B < 1) return PVMVMD_E_SHAPE;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;
    // the tensor-core products together in one persistent launch; every
    // other job takes the path pvmvmd_server_mvm gives it
    std::vector<BatchJob> grouped;
    std::vector<MvmJob> single;
    for (int i = 0; i < count; ++i) {
        const pvmvmd_mvm_batch_job &j = jobs[i];
        if (j.B > 1 && batched_grouped_eligible(j.W_dev, j.m, j.K, j.B)) {
            grouped.push_back(BatchJob{j.W_dev, j.Xhat_dev, j.Yhat_dev, j.m, j.K, j.B});
            continue;
        }
        if (j.B == 1) {
            MvmJob t{j.W_dev, j.Xhat_dev, j.Yhat_dev, j.m, j.K, (size_t)j.K, 0};
            if (multi_eligible(t)) {
                single.push_back(t);
                continue;
            }
        }
        const int st = pvmvmd_server_mvm(j.W_dev, j.m, j.K, j.Xhat_dev, j.B, j.Yhat_dev, stream);
        if (st != PVMVMD_OK) return st;
    }
    if (!single.empty()) PV_CUDA(launch_gemv_multi(single.data(), (int)single.size(), s));
    if (!grouped.empty()) PV_CUDA(launch_batched_grouped(grouped.data(), (int)grouped.size(), err, s));
    return PVMVMD_OK;
}

namespace pv {
namespace {
// The verification of a call: challenges e_q <- E_{t_y}^{N_y} shared by the
// B vectors, g_q = G_y e_q, u_q = e_q^T Q, and accept_b from x_hat_b and
// y_hat_b, all on stream cs.
// beside_decrypt: a decrypt of t_x rows per vector runs beside the chain
// (standard mode), so a large batch keeps its challenge clusters small; in
// boost mode the chain is the whole decode and gets the wider clusters.
int verify_chain(pvmvmd_ctx *ctx, const pvmvmd_key *challenge_key, const uint32_t *Xhat_dev,
                 const uint32_t *Yhat_dev, int B, int32_t *accept_dev, cudaStream_t cs, bool beside_decrypt) {
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;
    const CodeDev &d = ctx->gy;
    int C;
    uint32_t slice;
    size_t smem;
    if (syndrome_fused_plan(ctx->Ny, ctx->t_y, &C, &slice, &smem)) {
        PV_CUDA(launch_syndrome_fused(*challenge_key, kTagChallenge, 0, ctx->Ny, ctx->t_y,
                                      (uint32_t)ctx->ell, d.pi2inv, d.v2p, d.v1, d.pi1inv, d.pi2,
                                      d.v2m, d.v1pm, ctx->m, ctx->rate, ctx->chal, nullptr, ctx->g, cs, false,
                                      beside_decrypt && B >= kChallengeLargeBatch ? kSpreadChallenge
                                                                                 : kSpreadChallengeSmallBatch));
    } else {
        PV_CUDA(launch_sample_sparse(*challenge_key, kTagChallenge, 0, ctx->Ny, ctx->t_y, ctx->ell,
                                     ctx->chal, ctx->status_y, scan_status_words(ctx->Ny, ctx->ell), cs));
        PV_CUDA(launch_syndrome_scan(d.pi2inv, d.v2p, d.v1, ctx->Ny, ctx->chal, ctx->t_y, ctx->ell,
                                     ctx->Fy, ctx->status_y, err, cs));
        PV_CUDA(launch_syndrome_gather(d.pi1inv, ctx->m, ctx->rate, ctx->Fy, ctx->Ny, nullptr, ctx->g,
                                       ctx->ell, cs));
    }
    PV_CUDA(launch_verify_u(ctx->Q, ctx->K, ctx->chal, ctx->t_y, ctx->ell, ctx->u, cs));
    PV_CUDA(launch_check(Xhat_dev, ctx->K, Yhat_dev, ctx->m, ctx->g, ctx->u, (uint32_t)ctx->ell, B,
                         accept_dev, cs));
    return PVMVMD_OK;
}

bool overlaps(const void *a, const void *b, size_t bytes) {
    const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
    return x < y + bytes && y < x + bytes;
}

// Verify and decrypt: Y = Yhat - P e_x from st, or Y = Yhat - mask_out when
// mask_out is given (boost mode).  The verification depends on the key,
// x_hat and y_hat but not on Y, so it runs on the context's side stream
// while the decrypt streams P^T on the caller's stream; the caller's stream
// then waits for the side stream.  When Y overwrites Yhat the verification
// must read Yhat first, and both run in order on the caller's stream.
int decode_verify_batch(pvmvmd_ctx *ctx, const void *st_dev, const uint32_t *mask_out_dev,
                        const uint32_t *Xhat_dev, const uint32_t *Yhat_dev, int B,
                        const pvmvmd_key *challenge_key, uint32_t *Y_dev, int32_t *accept_dev,
                        cudaStream_t s) {
    const bool in_place = overlaps(Y_dev, Yhat_dev, (size_t)B * ctx->m * sizeof(uint32_t));
    const cudaStream_t cs = in_place ? s : ctx->side;
    if (!in_place) {
        PV_CUDA(cudaEventRecord(ctx->fork, s));
        PV_CUDA(cudaStreamWaitEvent(ctx->side, ctx->fork, 0));
    }
    int st = verify_chain(ctx, challenge_key, Xhat_dev, Yhat_dev, B, accept_dev, cs, mask_out_dev == nullptr);
    if (st) return st;
    PV_CUDA(launch_decrypt(ctx->PT, ctx->m, static_cast<const uint32_t *>(st_dev), ctx->t_x, (uint32_t)ctx->Nx,
                           Yhat_dev, B, Y_dev, s, mask_out_dev));
    if (!in_place) {
        PV_CUDA(cudaEventRecord(ctx->join, ctx->side));
        PV_CUDA(cudaStreamWaitEvent(s, ctx->join, 0));
    }
    return PVMVMD_OK;
}
}  // namespace
}  // namespace pv

int pvmvmd_decode_verify(pvmvmd_ctx *ctx, const void *st_dev, const uint32_t *Xhat_dev,
                         const uint32_t *Yhat_dev, int B, const pvmvmd_key *challenge_key,
                         uint32_t *Y_dev, int32_t *accept_dev, void *stream) {
    if (!ctx || !st_dev || !Xhat_dev || !Yhat_dev || !challenge_key || !Y_dev || !accept_dev)
        return PVMVMD_E_ARG;
    if (B < 1) return PVMVMD_E_SHAPE;
    return pv::decode_verify_batch(ctx, st_dev, nullptr, Xhat_dev, Yhat_dev, B, challenge_key, Y_dev,
                                   accept_dev, static_cast<cudaStream_t>(stream));
}

int pvmvmd_boost_decode_verify(pvmvmd_ctx *ctx, const uint32_t *mask_out_dev,
                               const uint32_t *Xhat_dev, const uint32_t *Yhat_dev, int B,
                               const pvmvmd_key *challenge_key, uint32_t *Y_dev,
                               int32_t *accept_dev, void *stream) {
    if (!ctx || !mask_out_dev || !Xhat_dev || !Yhat_dev || !challenge_key || !Y_dev || !accept_dev)
        return PVMVMD_E_ARG;
    if (B < 1) return PVMVMD_E_SHAPE;
    return pv::decode_verify_batch(ctx, nullptr, mask_out_dev, Xhat_dev, Yhat_dev, B, challenge_key,
                                   Y_dev, accept_dev, static_cast<cudaStream_t>(stream));
}

namespace pv {
namespace {
// Scratch of pvmvmd_code_encode_lanes: S (N x L), the scan's 64-bit status
// words and its ticket word, each at a 16-byte aligned offset.
struct EncodeScratch {
    size_t s_off, status_off, ticket_off, bytes;
};
EncodeScratch encode_scratch_layout(uint32_t N, uint32_t L) {
    auto up = [](size_t b) { return (b + 15) & ~(size_t)15; };
    EncodeScratch e;
    e.s_off = 0;
    e.status_off = up((size_t)N * L * 4);
    e.ticket_off = e.status_off + up(encode_scan_status_words(N, L) * 8);
    e.bytes = e.ticket_off + 16;
    return e;
}
}  // namespace
}  // namespace pv

int pvmvmd_code_encode_scratch(const pvmvmd_ctx *ctx, int which, int L, size_t *bytes) {
    if (!ctx || !bytes || (which != 0 && which != 1)) return PVMVMD_E_ARG;
    if (L < 1) return PVMVMD_E_SHAPE;
    const uint32_t N = which == 0 ? ctx->Nx : ctx->Ny;
    *bytes = pv::encode_scratch_layout(N, (uint32_t)L).bytes;
    return PVMVMD_OK;
}

int pvmvmd_code_encode_lanes(const pvmvmd_ctx *ctx, int which, const uint32_t *X_dev, int L,
                             uint32_t *Y_dev, void *scratch_dev, void *stream) {
    using namespace pv;
    if (!ctx || !X_dev || !Y_dev || !scratch_dev || (which != 0 && which != 1)) return PVMVMD_E_ARG;
    if (L < 1) return PVMVMD_E_SHAPE;
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;
    const CodeDev &d = which == 0 ? ctx->gx : ctx->gy;
    const uint32_t n = which == 0 ? (uint32_t)ctx->K : (uint32_t)ctx->m;
    const EncodeScratch lay = encode_scratch_layout(n * (uint32_t)ctx->rate, (uint32_t)L);
    uint8_t *base = static_cast<uint8_t *>(scratch_dev);
    return encode_lanes_into(d, n, (uint32_t)ctx->rate, X_dev, false, (size_t)L, (uint32_t)L, Y_dev, (size_t)L,
                             reinterpret_cast<uint32_t *>(base + lay.s_off),
                             reinterpret_cast<unsigned long long *>(base + lay.status_off),
                             reinterpret_cast<uint32_t *>(base + lay.ticket_off), err,
                             static_cast<cudaStream_t>(stream));
}

int pvmvmd_debug_expire_wait(int site, uint32_t index, uint64_t limit) {
    if (site != PVMVMD_DEBUG_WAIT_OFF && site != PVMVMD_DEBUG_WAIT_SCAN && site != PVMVMD_DEBUG_WAIT_PRODUCT)
        return PVMVMD_E_ARG;
    if (site != PVMVMD_DEBUG_WAIT_OFF && limit == 0) return PVMVMD_E_ARG;
    std::lock_guard<std::mutex> lock(g_debug_mu);
    g_debug.site = site;
    g_debug.index = site == PVMVMD_DEBUG_WAIT_OFF ? 0u : index;
    g_debug.limit = site == PVMVMD_DEBUG_WAIT_OFF ? 0u : limit;
    return PVMVMD_OK;
}

unsigned long long pvmvmd_kernel_launches(void) { return pv::kernel_launches(); }

int pvmvmd_device_status(void *stream) {
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) {
        (void)cudaGetLastError();
        return PVMVMD_E_CUDA;
    }
    return read_and_clear_error();
}

int pvmvmd_ctx_info(const pvmvmd_ctx *ctx, pvmvmd_ctx_view *v) {
    if (!ctx || !v) return PVMVMD_E_ARG;
    v->m = ctx->m;
    v->K = ctx->K;
    v->rate = ctx->rate;
    v->N_x = ctx->Nx;
    v->N_y = ctx->Ny;
    v->t_x = ctx->t_x;
    v->t_y = ctx->t_y;
    v->ell = ctx->ell;
    v->gx_pi1 = ctx->gx.pi1;
    v->gx_pi2 = ctx->gx.pi2;
    v->gx_v1 = ctx->gx.v1;
    v->gx_v2 = ctx->gx.v2;
    v->gy_pi1 = ctx->gy.pi1;
    v->gy_pi2 = ctx->gy.pi2;
    v->gy_v1 = ctx->gy.v1;
    v->gy_v2 = ctx->gy.v2;
    v->PT = ctx->PT;
    v->Q = ctx->Q;
    return PVMVMD_OK;
}

}  // extern "C"


// ---------------------------------------------------------------------------
// Batch verification, Protocol 2
// ---------------------------------------------------------------------------
void pvmvmd_bv_destroy(pvmvmd_bv_ctx *ctx) {
    if (!ctx) return;
    int cur = 0;
    cudaGetDevice(&cur);
    cudaSetDevice(ctx->device);
    for (void *p : ctx->owned) cudaFree(p);
    cudaSetDevice(cur);
    delete ctx;
}

int pvmvmd_bv_preprocess(const int8_t *W_dev, int B, int m, int n, const pvmvmd_bv_params *params,
                         const pvmvmd_key *key, void *stream, pvmvmd_bv_ctx **out) {
    using namespace pv;
    if (!out) return PVMVMD_E_ARG;
    *out = nullptr;
    if (!W_dev || !key) return PVMVMD_E_ARG;
    if (B < 1 || m < 1 || n < 1) return PVMVMD_E_SHAPE;
    const int rate = params && params->rate ? params->rate : 8;
    const long long N = (long long)rate * m, N2 = (long long)rate * B * n;
    // the device sampler holds a bitmap of N bits in shared memory
    if (rate < 2 || N > 8LL * PVMVMD_MAX_K || N2 > 8LL * PVMVMD_MAX_K) return PVMVMD_E_SHAPE;
    const int t = params && params->t ? params->t : 31, ell = params && params->ell ? params->ell : 2;
    const int t2 = params && params->t2 ? params->t2 : 31, ell2 = params && params->ell2 ? params->ell2 : 2;
    if (t < 1 || ell < 1 || t2 < 1 || ell2 < 1 || t > N || t2 > N2) return PVMVMD_E_PARAM;
    int st = check_device();
    if (st) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;
    pvmvmd_bv_ctx *c = new (std::nothrow) pvmvmd_bv_ctx();
    if (!c) return PVMVMD_E_NOMEM;
    cudaGetDevice(&c->device);
    c->B = B; c->m = m; c->n = n; c->rate = rate; c->N = (int)N; c->N2 = (int)N2;
    c->t = t; c->ell = ell; c->t2 = t2; c->ell2 = ell2;
    auto fail = [&](int code) {
        pvmvmd_bv_destroy(c);
        return code;
    };
    const uint32_t Bn = (uint32_t)B * n;
    if ((st = upload_code(c, c->g, *key, 3, (uint32_t)N, s))) return fail(st);
    if ((st = upload_code(c, c->g2, *key, 4, (uint32_t)N2, s))) return fail(st);
    const size_t sw = encode_scan_status_words((uint32_t)N, (uint32_t)B);
    if (ctx_alloc(c, &c->Qs, (size_t)N * Bn) != cudaSuccess ||
        ctx_alloc(c, &c->QauxT, (size_t)N2 * N) != cudaSuccess ||
        ctx_alloc(c, &c->Yt, (size_t)m * B) != cudaSuccess ||
        ctx_alloc(c, &c->Z, (size_t)N * B) != cudaSuccess ||
        ctx_alloc(c, &c->chal2, (size_t)ell2 * 2 * t2) != cudaSuccess ||
        ctx_alloc(c, &c->R, (size_t)ell2 * Bn) != cudaSuccess ||
        ctx_alloc(c, &c->F2, (size_t)ell2 * N2) != cudaSuccess ||
        ctx_alloc(c, &c->eS, (size_t)N * B) != cudaSuccess || ctx_alloc(c, &c->estatus, sw) != cudaSuccess ||
        ctx_alloc(c, &c->eticket, 1) != cudaSuccess ||
        ctx_alloc(c, &c->status, scan_status_words((uint32_t)N2, (uint32_t)ell2)) != cudaSuccess)
        return fail(PVMVMD_E_NOMEM);
    // Q_b = G^T M_b into the column block b n of Qs (the lanes are M_b's columns)
    for (int b = 0; b < B; ++b) {
        st = encode_lanes(c->g, (uint32_t)m, (uint32_t)rate, W_dev + (size_t)b * m * n, true, (size_t)n,
                          (uint32_t)n, c->Qs + (size_t)b * n, (size_t)Bn, err, s);
        if (st) return fail(st);
    }
    // Qaux = Qt^T G': row i is G'^T applied to row i of Qs; encode with the
    // N rows of Qs as lanes, so Qs is transposed first (Qt, B n x N)
    uint32_t *Qt = nullptr;
    if (dev_alloc(&Qt, (size_t)Bn * N) != cudaSuccess) return fail(PVMVMD_E_NOMEM);
    if (launch_transpose_u32(c->Qs, (int)N, (int)Bn, Qt, s) != cudaSuccess) {
        cudaFree(Qt);
        return fail(PVMVMD_E_CUDA);
    }
    st = encode_lanes(c->g2, Bn, (uint32_t)rate, Qt, false, (size_t)N, (uint32_t)N, c->QauxT, (size_t)N, err, s);
    cudaFree(Qt);
    if (st) return fail(st);
    if ((st = read_and_clear_error())) return fail(st);
    *out = c;
    return PVMVMD_OK;
}

int pvmvmd_bv_challenge(pvmvmd_bv_ctx *ctx, const pvmvmd_key *key, uint32_t *chal_dev, void *stream) {
    using namespace pv;
    if (!ctx || !key || !chal_dev) return PVMVMD_E_ARG;
    PV_CUDA(launch_sample_sparse(*key, kTagBvPrimary, 0, (uint32_t)ctx->N, (uint32_t)ctx->t,
                                 (uint32_t)ctx->ell, chal_dev, nullptr, 0, static_cast<cudaStream_t>(stream)));
    return PVMVMD_OK;
}

int pvmvmd_bv_server_project(const pvmvmd_bv_ctx *ctx, const uint32_t *chal_dev, uint32_t *u_dev,
                             void *stream) {
    using namespace pv;
    if (!ctx || !chal_dev || !u_dev) return PVMVMD_E_ARG;
    PV_CUDA(launch_verify_u(ctx->Qs, ctx->B * ctx->n, chal_dev, (uint32_t)ctx->t, (uint32_t)ctx->ell, u_dev,
                            static_cast<cudaStream_t>(stream)));
    return PVMVMD_OK;
}

int pvmvmd_bv_check(pvmvmd_bv_ctx *ctx, const uint32_t *X_dev, const uint32_t *Y_dev, const uint32_t *chal_dev,
                    const uint32_t *u_dev, const pvmvmd_key *key2, int32_t *accept_dev, void *stream) {
    using namespace pv;
    if (!ctx || !X_dev || !Y_dev || !chal_dev || !u_dev || !key2 || !accept_dev) return PVMVMD_E_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t *err = error_word();
    if (!err) return PVMVMD_E_CUDA;
    const uint32_t Bn = (uint32_t)ctx->B * ctx->n;
    // z_b = G^T y_b (the B outputs as lanes)
    PV_CUDA(launch_transpose_u32(Y_dev, ctx->B, ctx->m, ctx->Yt, s));
    int st = encode_lanes_into(ctx->g, (uint32_t)ctx->m, (uint32_t)ctx->rate, ctx->Yt, false, (size_t)ctx->B,
                               (uint32_t)ctx->B, ctx->Z, (size_t)ctx->B, ctx->eS, ctx->estatus, ctx->eticket,
                               err, s);
    if (st) return st;
    // secondary challenges, drawn after the responses, and r^(j) = G' e'^(j)
    const CodeDev &d = ctx->g2;
    int C;
    uint32_t slice;
    size_t smem;
    if (syndrome_fused_plan((uint32_t)ctx->N2, (uint32_t)ctx->t2, &C, &slice, &smem)) {
        PV_CUDA(launch_syndrome_fused(*key2, kTagBvSecondary, 0, (uint32_t)ctx->N2, (uint32_t)ctx->t2,
                                      (uint32_t)ctx->ell2, d.pi2inv, d.v2p, d.v1, d.pi1inv, d.pi2, d.v2m,
                                      d.v1pm, Bn, (uint32_t)ctx->rate, ctx->chal2, nullptr, ctx->R, s));
    } else {
        PV_CUDA(launch_sample_sparse(*key2, kTagBvSecondary, 0, (uint32_t)ctx->N2, (uint32_t)ctx->t2,
                                     (uint32_t)ctx->ell2, ctx->chal2, ctx->status,
                                     scan_status_words((uint32_t)ctx->N2, (uint32_t)ctx->ell2), s));
        PV_CUDA(launch_syndrome_scan(d.pi2inv, d.v2p, d.v1, (uint32_t)ctx->N2, ctx->chal2, (uint32_t)ctx->t2,
                                     (uint32_t)ctx->ell2, ctx->F2, ctx->status, err, s));
        PV_CUDA(launch_syndrome_gather(d.pi1inv, Bn, (uint32_t)ctx->rate, ctx->F2, (uint32_t)ctx->N2, nullptr,
                                       ctx->R, (uint32_t)ctx->ell2, s));
    }
    PV_CUDA(launch_bv_checks(ctx->QauxT, ctx->N, (int)Bn, ctx->n, ctx->B, chal_dev, (uint32_t)ctx->t,
                             (uint32_t)ctx->ell, ctx->chal2, (uint32_t)ctx->t2, (uint32_t)ctx->ell2, u_dev,
                             ctx->R, X_dev, ctx->Z, accept_dev, s));
    return PVMVMD_OK;
}

int pvmvmd_bv_info(const pvmvmd_bv_ctx *ctx, pvmvmd_bv_view *v) {
    if (!ctx || !v) return PVMVMD_E_ARG;
    v->B = ctx->B; v->m = ctx->m; v->n = ctx->n; v->rate = ctx->rate; v->N = ctx->N; v->N2 = ctx->N2;
    v->t = ctx->t; v->ell = ctx->ell; v->t2 = ctx->t2; v->ell2 = ctx->ell2;
    v->Qs = ctx->Qs;
    v->QauxT = ctx->QauxT;
    v->chal2 = ctx->chal2;
    return PVMVMD_OK;
}

