/*
 * pvMVMD oracle — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, exact CPU restatement of what the pvMVMD hot path computes
 * (Maverick, arXiv 2609.10264).  Only the test suite, the package smoke check
 * and the benchmark's CPU-baseline leg may load this file.  It shares no code
 * with the CUDA library: the random generator, the samplers, the RAA code, the
 * field arithmetic and every protocol step are written out here a second time,
 * in the most direct form the paper's definitions allow.
 *
 * Field: BabyBear, q = 15 * 2^27 + 1 (Sec. 7.1).  Every field element is a
 * uint32 in canonical form [0, q).  Arithmetic is done in uint64 with a
 * reduction after every single operation (no lazy reduction, no tricks).
 *
 * Randomness: the paper does not say how its Rust code draws random values.
 * The library and this oracle both implement one counter-based generator from
 * its published definition, the ChaCha20 block function of RFC 8439 Sec. 2.3,
 * and one sampler specification on top of it (stated at each function).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_Q 2013265921ULL

/* ---------------------------------------------------------------------- */
/* Field arithmetic over F_q (Sec. 7.1): one reduction per operation.      */
/* ---------------------------------------------------------------------- */
static uint64_t f_add(uint64_t a, uint64_t b) { return (a + b) % ORC_Q; }
static uint64_t f_sub(uint64_t a, uint64_t b) { return (a + ORC_Q - b) % ORC_Q; }
static uint64_t f_mul(uint64_t a, uint64_t b) { return (a * b) % ORC_Q; }
/* Embed a signed integer into F_q (the int8 weights of Sec. 7.2.1). */
static uint64_t f_lift(int64_t v) {
    int64_t r = v % (int64_t)ORC_Q;
    if (r < 0) r += (int64_t)ORC_Q;
    return (uint64_t)r;
}

/* Instrumentation: field operations performed by the RAA maps (App. B
 * counts at most 4N for an encoding and 5N for a syndrome).  Copies and
 * permutations are not field operations and are not counted. */
static uint64_t g_field_ops = 0;
uint64_t orc_field_ops(void) { return g_field_ops; }
void orc_reset_field_ops(void) { g_field_ops = 0; }
static uint64_t c_add(uint64_t a, uint64_t b) { g_field_ops++; return f_add(a, b); }
static uint64_t c_mul(uint64_t a, uint64_t b) { g_field_ops++; return f_mul(a, b); }

/* ---------------------------------------------------------------------- */
/* ChaCha20 block function, RFC 8439 Sec. 2.1-2.3.                          */
/* ---------------------------------------------------------------------- */
static uint32_t rotl32(uint32_t v, int c) { return (v << c) | (v >> (32 - c)); }

void orc_chacha_quarter_round(uint32_t *x, int a, int b, int c, int d) {
    x[a] += x[b]; x[d] ^= x[a]; x[d] = rotl32(x[d], 16);
    x[c] += x[d]; x[b] ^= x[c]; x[b] = rotl32(x[b], 12);
    x[a] += x[b]; x[d] ^= x[a]; x[d] = rotl32(x[d], 8);
    x[c] += x[d]; x[b] ^= x[c]; x[b] = rotl32(x[b], 7);
}

void orc_chacha20_block(const uint32_t key[8], uint32_t counter,
                        const uint32_t nonce[3], uint32_t out[16]) {
    uint32_t s[16], x[16];
    s[0] = 0x61707865u; s[1] = 0x3320646eu; s[2] = 0x79622d32u; s[3] = 0x6b206574u;
    for (int i = 0; i < 8; i++) s[4 + i] = key[i];
    s[12] = counter;
    s[13] = nonce[0]; s[14] = nonce[1]; s[15] = nonce[2];
    memcpy(x, s, sizeof s);
    for (int round = 0; round < 10; round++) {
        orc_chacha_quarter_round(x, 0, 4, 8, 12);
        orc_chacha_quarter_round(x, 1, 5, 9, 13);
        orc_chacha_quarter_round(x, 2, 6, 10, 14);
        orc_chacha_quarter_round(x, 3, 7, 11, 15);
        orc_chacha_quarter_round(x, 0, 5, 10, 15);
        orc_chacha_quarter_round(x, 1, 6, 11, 12);
        orc_chacha_quarter_round(x, 2, 7, 8, 13);
        orc_chacha_quarter_round(x, 3, 4, 9, 14);
    }
    for (int i = 0; i < 16; i++) out[i] = x[i] + s[i];
}

/* A stream is the ChaCha20 keystream for (key, nonce = (tag, idx_lo, idx_hi))
 * read as 32-bit words: word w is word (w mod 16) of block (w / 16). */
typedef struct {
    uint32_t key[8];
    uint32_t nonce[3];
    uint64_t pos;
    uint64_t have_block;
    uint32_t buf[16];
} orc_stream;

static void st_init(orc_stream *s, const uint32_t key[8], uint32_t tag, uint64_t idx) {
    memcpy(s->key, key, 8 * sizeof(uint32_t));
    s->nonce[0] = tag;
    s->nonce[1] = (uint32_t)idx;
    s->nonce[2] = (uint32_t)(idx >> 32);
    s->pos = 0;
    s->have_block = UINT64_MAX;
}

static uint32_t st_next(orc_stream *s) {
    uint64_t blk = s->pos / 16;
    if (blk != s->have_block) {
        orc_chacha20_block(s->key, (uint32_t)blk, s->nonce, s->buf);
        s->have_block = blk;
    }
    uint32_t w = s->buf[s->pos % 16];
    s->pos++;
    return w;
}

uint32_t orc_stream_word(const uint32_t key[8], uint32_t tag, uint64_t idx, uint64_t i) {
    uint32_t out[16], nonce[3] = {tag, (uint32_t)idx, (uint32_t)(idx >> 32)};
    orc_chacha20_block(key, (uint32_t)(i / 16), nonce, out);
    return out[i % 16];
}

static int bit_length(uint32_t v) {
    int b = 0;
    while (v) { b++; v >>= 1; }
    return b;
}

/* Uniform integer in [0, k): k <= 1 gives 0 and reads nothing; otherwise read
 * words, keep the top bit_length(k-1) bits, accept the first value below k. */
static uint32_t st_below(orc_stream *s, uint32_t k) {
    if (k <= 1) return 0;
    int b = bit_length(k - 1);
    for (;;) {
        uint32_t v = st_next(s) >> (32 - b);
        if (v < k) return v;
    }
}

/* Uniform element of F (nonzero = 0) or of F* (nonzero = 1): read words, keep
 * the top 31 bits, accept the first value in range. */
static uint32_t st_field(orc_stream *s, int nonzero) {
    for (;;) {
        uint32_t v = st_next(s) >> 1;
        if (v < ORC_Q && (!nonzero || v != 0)) return v;
    }
}

/* ---------------------------------------------------------------------- */
/* Samplers.                                                               */
/* ---------------------------------------------------------------------- */

/* Uniform permutation of [N]: Fisher-Yates from the last index down.
 * perm[j] = pi(j). */
void orc_sample_permutation(const uint32_t key[8], uint32_t tag, uint64_t idx,
                            uint32_t N, uint32_t *perm) {
    orc_stream s;
    st_init(&s, key, tag, idx);
    for (uint32_t i = 0; i < N; i++) perm[i] = i;
    for (uint32_t i = N; i-- > 1;) {
        uint32_t j = st_below(&s, i + 1);
        uint32_t t = perm[i]; perm[i] = perm[j]; perm[j] = t;
    }
}

/* N draws from F (nonzero = 0) or F* (nonzero = 1), in order. */
void orc_sample_field_vector(const uint32_t key[8], uint32_t tag, uint64_t idx,
                             uint32_t N, int nonzero, uint32_t *out) {
    orc_stream s;
    st_init(&s, key, tag, idx);
    for (uint32_t i = 0; i < N; i++) out[i] = st_field(&s, nonzero);
}

/* Uniform element of E_t^N (Sec. 3 notation; noise of App. A): a uniform
 * t-subset of [N] with values uniform in F*.  The support is the first t
 * distinct values of the sequence st_below(N) read from stream (tag, 2*idx);
 * it is returned in ascending order.  The k-th smallest support index gets
 * the k-th draw from F* of stream (tag, 2*idx + 1).  Returns -1 if t > N. */
int orc_sample_sparse(const uint32_t key[8], uint32_t tag, uint64_t idx,
                      uint32_t N, uint32_t t, uint32_t *support, uint32_t *values) {
    if (t > N) return -1;
    unsigned char *chosen = (unsigned char *)calloc(N ? N : 1, 1);
    if (!chosen) return -2;
    orc_stream s;
    st_init(&s, key, tag, 2 * idx);
    uint32_t have = 0;
    while (have < t) {
        uint32_t v = st_below(&s, N);
        if (!chosen[v]) { chosen[v] = 1; have++; }
    }
    uint32_t k = 0;
    for (uint32_t i = 0; i < N; i++)
        if (chosen[i]) support[k++] = i;
    free(chosen);
    orc_stream sv;
    st_init(&sv, key, tag, 2 * idx + 1);
    for (uint32_t j = 0; j < t; j++) values[j] = st_field(&sv, 1);
    return 0;
}

/* Domain tags.  G_x (privacy code) uses 1..4, G_y (verification code) 5..8. */
enum { TAG_PI1 = 1, TAG_PI2 = 2, TAG_V1 = 3, TAG_V2 = 4, TAG_MASK = 9, TAG_CHALLENGE = 10 };

/* RAA generator G = R Pi1 V1 A Pi2 V2 A (App. B): sample pi1, pi2 uniform
 * permutations of [N] and v1, v2 uniform in (F*)^N.  which = 0 for G_x,
 * which = 1 for G_y. */
void orc_code_sample(const uint32_t key[8], int which, uint32_t N,
                     uint32_t *pi1, uint32_t *pi2, uint32_t *v1, uint32_t *v2) {
    uint32_t base = 4u * (uint32_t)which;  /* code `which` reads tags 4 which + 1 .. 4 which + 4 */
    orc_sample_permutation(key, base + TAG_PI1, 0, N, pi1);
    orc_sample_permutation(key, base + TAG_PI2, 0, N, pi2);
    orc_sample_field_vector(key, base + TAG_V1, 0, N, 1, v1);
    orc_sample_field_vector(key, base + TAG_V2, 0, N, 1, v2);
}

/* ---------------------------------------------------------------------- */
/* RAA maps, App. B: each component matrix applied as its own stage, in the */
/* order of the composition, on dense length-N arrays.                      */
/*   R_{i,j} = 1 iff (i-1) r < j <= i r     (repetition, n x N)             */
/*   Pi_{i,j} = 1 iff pi(j) = i             (permutation)                   */
/*   V = diag(v)                            (randomisation)                 */
/*   A_{i,j} = 1 iff i <= j                 (accumulation, upper triangle)  */
/* ---------------------------------------------------------------------- */

/* Encoding w -> G^T w = A^T V2 Pi2^T A^T V1 Pi1^T R^T w (w in F^n, out in F^N). */
void orc_raa_encode(uint32_t n, uint32_t r, const uint32_t *pi1, const uint32_t *pi2,
                    const uint32_t *v1, const uint32_t *v2, const uint32_t *w, uint32_t *out) {
    uint64_t N = (uint64_t)n * r;
    uint64_t *a = (uint64_t *)malloc(N * sizeof(uint64_t));
    uint64_t *b = (uint64_t *)malloc(N * sizeof(uint64_t));
    /* R^T w: (R^T w)_j = w_i for the i with (i-1) r < j <= i r. */
    for (uint64_t j = 0; j < N; j++) a[j] = w[j / r];
    /* Pi1^T: (Pi^T u)_j = sum_i Pi_{i,j} u_i = u_{pi(j)}. */
    for (uint64_t j = 0; j < N; j++) b[j] = a[pi1[j]];
    /* V1. */
    for (uint64_t j = 0; j < N; j++) b[j] = c_mul(v1[j], b[j]);
    /* A^T: (A^T u)_j = sum_{i <= j} u_i, a prefix sum. */
    for (uint64_t j = 1; j < N; j++) b[j] = c_add(b[j - 1], b[j]);
    /* Pi2^T. */
    for (uint64_t j = 0; j < N; j++) a[j] = b[pi2[j]];
    /* V2. */
    for (uint64_t j = 0; j < N; j++) a[j] = c_mul(v2[j], a[j]);
    /* A^T. */
    for (uint64_t j = 1; j < N; j++) a[j] = c_add(a[j - 1], a[j]);
    for (uint64_t j = 0; j < N; j++) out[j] = (uint32_t)a[j];
    free(a);
    free(b);
}

/* Syndrome v -> G v = R Pi1 V1 A Pi2 V2 A v (v in F^N, out in F^n). */
void orc_raa_syndrome(uint32_t n, uint32_t r, const uint32_t *pi1, const uint32_t *pi2,
                      const uint32_t *v1, const uint32_t *v2, const uint32_t *v, uint32_t *out) {
    uint64_t N = (uint64_t)n * r;
    uint64_t *a = (uint64_t *)malloc(N * sizeof(uint64_t));
    uint64_t *b = (uint64_t *)malloc(N * sizeof(uint64_t));
    for (uint64_t j = 0; j < N; j++) a[j] = v[j];
    /* A: (A u)_i = sum_{j >= i} u_j, a suffix sum. */
    for (uint64_t j = N - 1; j-- > 0;) a[j] = c_add(a[j], a[j + 1]);
    /* V2. */
    for (uint64_t j = 0; j < N; j++) a[j] = c_mul(v2[j], a[j]);
    /* Pi2: (Pi u)_i = sum_j Pi_{i,j} u_j, i.e. entry j moves to pi(j). */
    for (uint64_t j = 0; j < N; j++) b[pi2[j]] = a[j];
    /* A. */
    for (uint64_t j = N - 1; j-- > 0;) b[j] = c_add(b[j], b[j + 1]);
    /* V1. */
    for (uint64_t j = 0; j < N; j++) b[j] = c_mul(v1[j], b[j]);
    /* Pi1. */
    for (uint64_t j = 0; j < N; j++) a[pi1[j]] = b[j];
    /* R: (R u)_i = sum of the i-th block of r consecutive entries. */
    for (uint64_t i = 0; i < n; i++) {
        uint64_t acc = a[i * r];
        for (uint64_t c = 1; c < r; c++) acc = c_add(acc, a[i * r + c]);
        out[i] = (uint32_t)acc;
    }
    free(a);
    free(b);
}

/* ---------------------------------------------------------------------- */
/* Parameters (Eq. 1 of Sec. 6.2, Thm 5.2 and its proof, Sec. 7.1).           */
/* ---------------------------------------------------------------------- */

/* Mask sparsity, Eq. (1): smallest integer t with t >= ln2 (lambda - log2 N)/delta. */
int orc_t_x(int lambda, double N, double delta) {
    return (int)ceil(log(2.0) * ((double)lambda - log2(N)) / delta);
}

/* Verification parameters from Thm 5.2 and the two cases of its proof.
 * Case 1 (1/(|F|-1) <= 2^-(kappa+1)): ell = 1 and (1-delta)^t <= 2^-(kappa+1).
 * Case 2 (otherwise): (1-delta)^t <= 1/(|F|-1) and
 *   ell = ceil(kappa / (log2(|F|-1) - 1)).
 * t_thm is the theorem's stated formula, which uses max(log2(|F|-1), kappa+1)
 * in both cases. */
void orc_verify_params(int kappa, double delta, int *t_case, int *t_thm, int *ell) {
    double lf = log2((double)(ORC_Q - 1));
    double per = -log2(1.0 - delta);
    *t_thm = (int)ceil((lf > kappa + 1 ? lf : (double)(kappa + 1)) / per);
    *ell = (int)ceil((double)kappa / (lf - 1.0));
    if (lf >= kappa + 1) {
        *t_case = (int)ceil((double)(kappa + 1) / per);
        *ell = 1;
    } else {
        *t_case = (int)ceil(lf / per);
    }
}

/* ---------------------------------------------------------------------- */
/* Server MVM, y_hat = M x_hat over F_q (Sec. 6.1; server's only online work).*/
/* Textbook: lift each weight, one multiply and one add per MAC, each reduced.*/
/* ---------------------------------------------------------------------- */
void orc_server_mvm_rows(const int8_t *W, uint32_t m, uint32_t K, const uint32_t *xhat,
                         const uint32_t *rows, uint32_t nrows, uint32_t *yhat) {
    (void)m;
    for (uint32_t t = 0; t < nrows; t++) {
        uint64_t i = rows[t];
        uint64_t acc = 0;
        for (uint64_t k = 0; k < K; k++)
            acc = f_add(acc, f_mul(f_lift(W[i * K + k]), xhat[k]));
        yhat[t] = (uint32_t)acc;
    }
}

void orc_server_mvm(const int8_t *W, uint32_t m, uint32_t K, const uint32_t *xhat,
                    uint32_t *yhat) {
    for (uint64_t i = 0; i < m; i++) {
        uint64_t acc = 0;
        for (uint64_t k = 0; k < K; k++)
            acc = f_add(acc, f_mul(f_lift(W[i * K + k]), xhat[k]));
        yhat[i] = (uint32_t)acc;
    }
}

/* ---------------------------------------------------------------------- */
/* Protocol 3 (Pi_pvMVMD).                                                 */
/* ---------------------------------------------------------------------- */

/* Preprocess, P = M G_x: P^T = G_x^T M^T is m encodings of the rows of M
 * (Sec. 6.3).  Stored as P^T, row-major N_x x m. */
void orc_preprocess_PT(const int8_t *W, uint32_t m, uint32_t n, uint32_t r,
                       const uint32_t *pi1, const uint32_t *pi2, const uint32_t *v1,
                       const uint32_t *v2, uint32_t *PT) {
    uint64_t N = (uint64_t)n * r;
    uint32_t *row = (uint32_t *)malloc((size_t)n * sizeof(uint32_t));
    uint32_t *enc = (uint32_t *)malloc(N * sizeof(uint32_t));
    for (uint64_t i = 0; i < m; i++) {
        for (uint64_t k = 0; k < n; k++) row[k] = (uint32_t)f_lift(W[i * n + k]);
        orc_raa_encode(n, r, pi1, pi2, v1, v2, row, enc);
        for (uint64_t j = 0; j < N; j++) PT[j * m + i] = enc[j];
    }
    free(row);
    free(enc);
}

/* Preprocess, Q = G_y^T M: n encodings of the columns of M (Sec. 6.3).
 * Stored row-major N_y x n. */
void orc_preprocess_Q(const int8_t *W, uint32_t m, uint32_t n, uint32_t r,
                      const uint32_t *pi1, const uint32_t *pi2, const uint32_t *v1,
                      const uint32_t *v2, uint32_t *Qm) {
    uint64_t N = (uint64_t)m * r;
    uint32_t *col = (uint32_t *)malloc((size_t)m * sizeof(uint32_t));
    uint32_t *enc = (uint32_t *)malloc(N * sizeof(uint32_t));
    for (uint64_t k = 0; k < n; k++) {
        for (uint64_t i = 0; i < m; i++) col[i] = (uint32_t)f_lift(W[i * n + k]);
        orc_raa_encode(m, r, pi1, pi2, v1, v2, col, enc);
        for (uint64_t j = 0; j < N; j++) Qm[j * n + k] = enc[j];
    }
    free(col);
    free(enc);
}

/* Encrypt: e_x <- E_{t_x}^{N_x} (vector number b of the call), x' = G_x e_x,
 * x_hat = x + x', st = e_x.  Returns -1 if t_x > N_x. */
int orc_encrypt(uint32_t n, uint32_t r, const uint32_t *pi1, const uint32_t *pi2,
                const uint32_t *v1, const uint32_t *v2, const uint32_t key[8],
                uint64_t b, uint32_t t_x, const uint32_t *x, uint32_t *xhat,
                uint32_t *support, uint32_t *values) {
    uint64_t N = (uint64_t)n * r;
    if (orc_sample_sparse(key, TAG_MASK, b, (uint32_t)N, t_x, support, values)) return -1;
    uint32_t *e = (uint32_t *)calloc(N, sizeof(uint32_t));
    uint32_t *xp = (uint32_t *)malloc((size_t)n * sizeof(uint32_t));
    for (uint32_t j = 0; j < t_x; j++) e[support[j]] = values[j];
    orc_raa_syndrome(n, r, pi1, pi2, v1, v2, e, xp);
    for (uint64_t i = 0; i < n; i++) xhat[i] = (uint32_t)f_add(x[i], xp[i]);
    free(e);
    free(xp);
    return 0;
}

/* Verify, literally: z = G_y^T y_hat; for each of ell repetitions sample
 * e <- E_{t_y}^{N_y} (repetition number rep of the call), v_L = (e^T Q) x_hat,
 * v_R = e^T z; reject on the first mismatch.  Returns 1 accept, 0 reject,
 * -1 on bad parameters. */
int orc_verify(uint32_t m, uint32_t n, uint32_t r, const uint32_t *pi1, const uint32_t *pi2,
               const uint32_t *v1, const uint32_t *v2, const uint32_t *Qm,
               const uint32_t key[8], uint32_t t_y, uint32_t ell,
               const uint32_t *xhat, const uint32_t *yhat) {
    uint64_t N = (uint64_t)m * r;
    if (t_y > N) return -1;
    uint32_t *z = (uint32_t *)malloc(N * sizeof(uint32_t));
    uint32_t *supp = (uint32_t *)malloc((size_t)t_y * sizeof(uint32_t));
    uint32_t *vals = (uint32_t *)malloc((size_t)t_y * sizeof(uint32_t));
    uint64_t *eQ = (uint64_t *)malloc((size_t)n * sizeof(uint64_t));
    orc_raa_encode(m, r, pi1, pi2, v1, v2, yhat, z);
    int accept = 1;
    for (uint32_t rep = 0; rep < ell && accept; rep++) {
        orc_sample_sparse(key, TAG_CHALLENGE, rep, (uint32_t)N, t_y, supp, vals);
        for (uint64_t k = 0; k < n; k++) eQ[k] = 0;
        for (uint32_t j = 0; j < t_y; j++)
            for (uint64_t k = 0; k < n; k++)
                eQ[k] = f_add(eQ[k], f_mul(vals[j], Qm[(uint64_t)supp[j] * n + k]));
        uint64_t vL = 0, vR = 0;
        for (uint64_t k = 0; k < n; k++) vL = f_add(vL, f_mul(eQ[k], xhat[k]));
        for (uint32_t j = 0; j < t_y; j++) vR = f_add(vR, f_mul(vals[j], z[supp[j]]));
        if (vL != vR) accept = 0;
    }
    free(z); free(supp); free(vals); free(eQ);
    return accept;
}

/* Verify without the preprocessed Q, for matrices whose Q does not fit in host
 * memory: e^T Q = e^T G_y^T M = (G_y e)^T M by the definition of Q, so
 * v_L = ((G_y e)^T M) x_hat.  v_R is computed exactly as in orc_verify. */
int orc_verify_noQ(const int8_t *W, uint32_t m, uint32_t n, uint32_t r,
                   const uint32_t *pi1, const uint32_t *pi2, const uint32_t *v1,
                   const uint32_t *v2, const uint32_t key[8], uint32_t t_y, uint32_t ell,
                   const uint32_t *xhat, const uint32_t *yhat) {
    uint64_t N = (uint64_t)m * r;
    if (t_y > N) return -1;
    uint32_t *z = (uint32_t *)malloc(N * sizeof(uint32_t));
    uint32_t *e = (uint32_t *)malloc(N * sizeof(uint32_t));
    uint32_t *g = (uint32_t *)malloc((size_t)m * sizeof(uint32_t));
    uint32_t *supp = (uint32_t *)malloc((size_t)t_y * sizeof(uint32_t));
    uint32_t *vals = (uint32_t *)malloc((size_t)t_y * sizeof(uint32_t));
    uint64_t *eQ = (uint64_t *)malloc((size_t)n * sizeof(uint64_t));
    orc_raa_encode(m, r, pi1, pi2, v1, v2, yhat, z);
    int accept = 1;
    for (uint32_t rep = 0; rep < ell && accept; rep++) {
        orc_sample_sparse(key, TAG_CHALLENGE, rep, (uint32_t)N, t_y, supp, vals);
        memset(e, 0, N * sizeof(uint32_t));
        for (uint32_t j = 0; j < t_y; j++) e[supp[j]] = vals[j];
        orc_raa_syndrome(m, r, pi1, pi2, v1, v2, e, g);
        for (uint64_t k = 0; k < n; k++) eQ[k] = 0;
        for (uint64_t i = 0; i < m; i++)
            for (uint64_t k = 0; k < n; k++)
                eQ[k] = f_add(eQ[k], f_mul(g[i], f_lift(W[i * n + k])));
        uint64_t vL = 0, vR = 0;
        for (uint64_t k = 0; k < n; k++) vL = f_add(vL, f_mul(eQ[k], xhat[k]));
        for (uint32_t j = 0; j < t_y; j++) vR = f_add(vR, f_mul(vals[j], z[supp[j]]));
        if (vL != vR) accept = 0;
    }
    free(z); free(e); free(g); free(supp); free(vals); free(eQ);
    return accept;
}

/* Decrypt: y = y_hat - P e_x = y_hat - sum_{j in supp} e_j P_{:,j}, with P
 * stored as P^T (N_x x m), so column j of P is row j of P^T. */
void orc_decrypt(uint32_t m, const uint32_t *PT, uint32_t t_x, const uint32_t *support,
                 const uint32_t *values, const uint32_t *yhat, uint32_t *y) {
    for (uint64_t i = 0; i < m; i++) {
        uint64_t pe = 0;
        for (uint32_t j = 0; j < t_x; j++)
            pe = f_add(pe, f_mul(values[j], PT[(uint64_t)support[j] * m + i]));
        y[i] = (uint32_t)f_sub(yhat[i], pe);
    }
}

/* Decrypt of selected output rows when P^T is not held: column i of P^T is
 * the encoding G_x^T M_{i,:} of row i of M, so (P e_x)_i is read from it. */
void orc_decrypt_rows(const int8_t *W, uint32_t n, uint32_t r, const uint32_t *pi1,
                      const uint32_t *pi2, const uint32_t *v1, const uint32_t *v2,
                      uint32_t t_x, const uint32_t *support, const uint32_t *values,
                      const uint32_t *rows, uint32_t nrows, const uint32_t *yhat_rows,
                      uint32_t *y_rows) {
    uint64_t N = (uint64_t)n * r;
    uint32_t *row = (uint32_t *)malloc((size_t)n * sizeof(uint32_t));
    uint32_t *enc = (uint32_t *)malloc(N * sizeof(uint32_t));
    for (uint32_t t = 0; t < nrows; t++) {
        uint64_t i = rows[t];
        for (uint64_t k = 0; k < n; k++) row[k] = (uint32_t)f_lift(W[i * n + k]);
        orc_raa_encode(n, r, pi1, pi2, v1, v2, row, enc);
        uint64_t pe = 0;
        for (uint32_t j = 0; j < t_x; j++) pe = f_add(pe, f_mul(values[j], enc[support[j]]));
        y_rows[t] = (uint32_t)f_sub(yhat_rows[t], pe);
    }
    free(row);
    free(enc);
}
