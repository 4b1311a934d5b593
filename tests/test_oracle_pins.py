"""Pins for the oracle: checks against what the paper and mathematics fix.

Each test compares the oracle with something other than itself: values the
paper prints, published test vectors of the generator, dense matrices built
from the App. B component definitions, Python big-integer brute force,
algebraic identities, and the Lemma 5.1 acceptance probability.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from oracle import Q

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# --------------------------------------------------------------------------- generator

def test_chacha20_rfc8439_vectors():
    g = _golden("chacha20_rfc8439.json")
    qr = g["quarter_round_2_1_1"]
    out = oracle.chacha_quarter_round([int(v, 16) for v in qr["input"]], 0, 1, 2, 3)
    assert [int(v) for v in out] == [int(v, 16) for v in qr["output"]]
    blk = g["block_2_3_2"]
    kb = bytes.fromhex(blk["key_bytes"])
    nb = bytes.fromhex(blk["nonce_bytes"])
    key = np.frombuffer(kb, dtype="<u4").astype(np.uint32)
    nonce = np.frombuffer(nb, dtype="<u4").astype(np.uint32)
    out = oracle.chacha20_block(key, blk["counter"], nonce)
    assert [int(v) for v in out] == [int(v, 16) for v in blk["output_words"]]


def test_sampler_golden_seed0_unchanged():
    g = _golden("sampler_seed0.json")
    key = oracle.key_from_seed(0)
    assert [oracle.stream_word(key, 1, 0, i) for i in range(20)] == g["stream_words_tag1_idx0"]
    assert oracle.sample_permutation(key, 1, 0, 16).tolist() == g["perm_tag1_N16"]
    assert oracle.sample_field_vector(key, 3, 0, 8, True).tolist() == g["field_star_tag3_N8"]
    s, v = oracle.sample_sparse(key, oracle.TAG_MASK, 0, 2048, 12)
    assert s.tolist() == g["sparse_mask_b0_N2048_t12"]["support"]
    assert v.tolist() == g["sparse_mask_b0_N2048_t12"]["values"]


def test_stream_words_are_chacha_blocks():
    # word i of stream (tag, idx) is word i%16 of block i/16 with nonce (tag, idx_lo, idx_hi)
    key = oracle.key_from_seed(12345)
    idx = (7 << 32) | 3
    blk = oracle.chacha20_block(key, 2, [5, 3, 7])
    assert [oracle.stream_word(key, 5, idx, 32 + j) for j in range(16)] == [int(b) for b in blk]


# --------------------------------------------------------------------------- samplers

def test_permutation_is_uniform_small():
    # all 3! permutations of [3] appear with frequency ~1/6 over many keys
    counts = {}
    trials = 6000
    for s in range(trials):
        p = tuple(oracle.sample_permutation(oracle.key_from_seed(s), 1, 0, 3).tolist())
        counts[p] = counts.get(p, 0) + 1
    assert len(counts) == 6
    chi2 = sum((c - trials / 6) ** 2 / (trials / 6) for c in counts.values())
    assert chi2 < 25.7  # chi-square, 5 dof, p ~ 1e-4


def test_permutation_is_bijection_large():
    p = oracle.sample_permutation(oracle.key_from_seed(9), 2, 0, 100003)
    assert np.array_equal(np.sort(p), np.arange(100003, dtype=np.uint32))


def test_field_samples_in_range_and_uniform():
    v = oracle.sample_field_vector(oracle.key_from_seed(1), 3, 0, 200000, True)
    assert v.min() >= 1 and v.max() < Q
    hist = np.bincount((v.astype(np.uint64) * 16 // Q).astype(np.int64), minlength=16)
    exp = len(v) / 16
    assert ((hist - exp) ** 2 / exp).sum() < 45  # 15 dof


def test_sparse_support_and_values():
    N, t = 2048, 163
    hits = np.zeros(N)
    for s in range(400):
        supp, vals = oracle.sample_sparse(oracle.key_from_seed(s), oracle.TAG_MASK, s % 5, N, t)
        assert len(supp) == t and np.all(np.diff(supp.astype(np.int64)) > 0)
        assert supp.max() < N
        assert vals.min() >= 1 and vals.max() < Q
        hits[supp] += 1
    # each position is in the support with probability t/N
    coarse = hits.reshape(16, -1).sum(1)
    exp = 400 * t / 16
    assert ((coarse - exp) ** 2 / exp).sum() < 45


def test_sparse_full_support():
    supp, vals = oracle.sample_sparse(oracle.key_from_seed(3), 10, 0, 40, 40)
    assert supp.tolist() == list(range(40))
    with pytest.raises(ValueError):
        oracle.sample_sparse(oracle.key_from_seed(3), 10, 0, 40, 41)


# --------------------------------------------------------------------------- parameters

def test_paper_parameters():
    g = _golden("paper_params.json")
    assert Q == g["q"]["value"] == 15 * 2 ** 27 + 1
    for n, t in zip(g["t_x_by_n"]["n"], g["t_x_by_n"]["t_x"]):
        assert oracle.t_x(n) == t, (n, t)
    t_case, t_thm, ell = oracle.verify_params()
    assert t_case == g["t_y"]["value"]
    assert ell == g["ell"]["value"]
    # the theorem's stated formula, max(log2(|F|-1), kappa+1)/1, gives 41
    assert t_thm == 41


def test_paper_parameters_bound():
    # Thm 5.2 proof, Case 2: ((1-delta)^t + 1/(|F|-1))^ell <= 2^-kappa at t=31, ell=2
    eps = 0.5 ** 31 + 1.0 / (Q - 1)
    assert eps ** 2 <= 2.0 ** -40
    assert math.log2(eps ** 2) < -59.8


# --------------------------------------------------------------------------- RAA code

def _dense_components(code):
    """The App. B component matrices, built entry by entry from their
    definitions (1-indexed in the paper, 0-indexed here), as Python ints."""
    n, r, N = code.n, code.r, code.N
    R = [[1 if i * r <= j < (i + 1) * r else 0 for j in range(N)] for i in range(n)]

    def perm(p):
        return [[1 if int(p[j]) == i else 0 for j in range(N)] for i in range(N)]

    def diag(v):
        return [[int(v[i]) if i == j else 0 for j in range(N)] for i in range(N)]

    A = [[1 if i <= j else 0 for j in range(N)] for i in range(N)]
    return R, perm(code.pi1), diag(code.v1), A, perm(code.pi2), diag(code.v2)


def _mm(X, Y):
    return [[sum(X[i][k] * Y[k][j] for k in range(len(Y))) % Q for j in range(len(Y[0]))]
            for i in range(len(X))]


def _dense_G(code):
    R, P1, V1, A, P2, V2 = _dense_components(code)
    G = R
    for M in (P1, V1, A, P2, V2, A):
        G = _mm(G, M)
    return G


@pytest.mark.parametrize("n", [1, 2, 3, 4, 8])
def test_raa_matches_dense_definition(n):
    code = oracle.Code.sample(oracle.key_from_seed(100 + n), n % 2, n, 8)
    G = _dense_G(code)
    rng = np.random.default_rng(n)
    w = rng.integers(0, Q, n)
    v = rng.integers(0, Q, code.N)
    enc = [sum(G[i][j] * int(w[i]) for i in range(n)) % Q for j in range(code.N)]
    syn = [sum(G[i][j] * int(v[j]) for j in range(code.N)) % Q for i in range(n)]
    assert code.encode(w).tolist() == enc
    assert code.syndrome(v).tolist() == syn


def test_raa_other_rate_matches_dense():
    code = oracle.Code.sample(oracle.key_from_seed(7), 0, 5, 3)
    G = _dense_G(code)
    w = np.arange(1, 6)
    assert code.encode(w).tolist() == [sum(G[i][j] * int(w[i]) for i in range(5)) % Q
                                       for j in range(15)]


def test_raa_adjoint_identity():
    # <G^T w, v> = <w, G v> for every w, v
    code = oracle.Code.sample(oracle.key_from_seed(5), 1, 512, 8)
    rng = np.random.default_rng(0)
    for _ in range(3):
        w = rng.integers(0, Q, code.n)
        v = rng.integers(0, Q, code.N)
        lhs = sum(int(a) * int(b) for a, b in zip(code.encode(w), v)) % Q
        rhs = sum(int(a) * int(b) for a, b in zip(w, code.syndrome(v))) % Q
        assert lhs == rhs


def test_raa_linearity_and_unit_weight():
    code = oracle.Code.sample(oracle.key_from_seed(11), 0, 256, 8)
    rng = np.random.default_rng(1)
    a, b = rng.integers(0, Q, 256), rng.integers(0, Q, 256)
    ea, eb, eab = code.encode(a), code.encode(b), code.encode((a + b) % Q)
    assert np.array_equal((ea.astype(np.uint64) + eb) % Q, eab)
    # empirical distance check on the test code (not a guarantee; App. B)
    for k in range(0, 256, 37):
        u = np.zeros(256, np.uint32)
        u[k] = 1
        assert np.count_nonzero(code.encode(u)) >= code.N // 2


def test_raa_operation_counts():
    # App. B: at most 4N field operations per encoding, 5N per syndrome
    code = oracle.Code.sample(oracle.key_from_seed(2), 0, 1000, 8)
    oracle.reset_field_ops()
    code.encode(np.ones(code.n))
    assert oracle.field_ops() <= 4 * code.N
    oracle.reset_field_ops()
    code.syndrome(np.ones(code.N))
    assert oracle.field_ops() <= 5 * code.N


# --------------------------------------------------------------------------- server MVM

@pytest.mark.parametrize("shape", [(4, 4), (5, 7), (16, 16), (33, 64), (64, 64)])
def test_server_mvm_bruteforce(shape):
    m, K = shape
    rng = np.random.default_rng(m * 100 + K)
    W = rng.integers(-127, 128, (m, K)).astype(np.int8)
    x = rng.integers(0, Q, K).astype(np.uint32)
    ref = [sum(int(W[i, k]) * int(x[k]) for k in range(K)) % Q for i in range(m)]
    assert oracle.server_mvm(W, x).tolist() == ref
    rows = [0, m - 1, m // 2]
    assert oracle.server_mvm_rows(W, x, rows).tolist() == [ref[i] for i in rows]


@pytest.mark.parametrize("shape", [(4, 4, 1), (5, 7, 3), (33, 64, 5), (9, 300, 2)])
def test_server_mvm_batch_bruteforce(shape):
    """The batched oracle product against Python big integers, with the
    extremes of both operands in every vector."""
    m, K, B = shape
    rng = np.random.default_rng(m * 1000 + K + B)
    W = rng.integers(-128, 128, (m, K)).astype(np.int8)
    W[0] = -128
    X = rng.integers(0, Q, (B, K)).astype(np.uint32)
    X[:, 0] = Q - 1
    X[0] = (Q + 1) // 2
    ref = [[sum(int(W[i, k]) * int(X[b, k]) for k in range(K)) % Q for i in range(m)] for b in range(B)]
    assert oracle.server_mvm_batch(W, X).tolist() == ref


@pytest.mark.parametrize("m,K,B,block", [(70, 1000, 6, 4096), (300, 2048, 4, 64), (5, 131071, 2, 4096)])
def test_server_mvm_batch_matches_per_mac_loop(m, K, B, block):
    """The batched product equals the per-MAC C loop (itself pinned by brute
    force), up to the largest K the library accepts, over row blocks, with
    every weight at -128 or 127 and every x_hat at q - 1 or (q + 1) / 2 in
    some rows and vectors (the largest float64 partial sums)."""
    rng = np.random.default_rng(m + K + B)
    W = rng.integers(-128, 128, (m, K)).astype(np.int8)
    W[0] = -128
    W[1] = 127
    X = rng.integers(0, Q, (B, K)).astype(np.uint32)
    X[0] = Q - 1
    X[1] = (Q + 1) // 2
    got = oracle.server_mvm_batch(W, X, row_block=block)
    for b in range(B):
        assert np.array_equal(got[b], oracle.server_mvm(W, X[b])), b


def test_server_mvm_extremes_and_special_cases():
    K = 300
    W = np.full((3, K), -128, np.int8)
    W[1] = 127
    W[2, ::2] = -127
    x = np.full(K, Q - 1, np.uint32)
    ref = [sum(int(W[i, k]) * (Q - 1) for k in range(K)) % Q for i in range(3)]
    assert oracle.server_mvm(W, x).tolist() == ref
    rng = np.random.default_rng(3)
    W = rng.integers(-127, 128, (20, 20)).astype(np.int8)
    # identity weights return x_hat
    xh = rng.integers(0, Q, 20).astype(np.uint32)
    assert np.array_equal(oracle.server_mvm(np.eye(20, dtype=np.int8), xh), xh)
    # a unit vector returns the lifted column
    e = np.zeros(20, np.uint32)
    e[7] = 1
    assert np.array_equal(oracle.server_mvm(W, e), oracle.lift(W[:, 7]))
    # linearity of the masked product
    a, b = rng.integers(0, Q, 20), rng.integers(0, Q, 20)
    lhs = oracle.server_mvm(W, (a + b) % Q)
    rhs = (oracle.server_mvm(W, a).astype(np.uint64) + oracle.server_mvm(W, b)) % Q
    assert np.array_equal(lhs, rhs)


# --------------------------------------------------------------------------- protocol

@pytest.fixture(scope="module")
def tiny_pp():
    """A 256 x 256 int8 matrix, uniform in [-127, 127], the paper's parameters."""
    rng = np.random.default_rng(0)
    W = rng.integers(-127, 128, (256, 256)).astype(np.int8)
    return oracle.PublicParams(W, oracle.key_from_seed(0))


def test_preprocess_tables_are_encodings(tiny_pp):
    pp = tiny_pp
    i, k = 17, 200
    assert np.array_equal(pp.PT[:, i], pp.Gx.encode(oracle.lift(pp.W[i])))
    assert np.array_equal(pp.Q[:, k], pp.Gy.encode(oracle.lift(pp.W[:, k])))
    # P = M G_x: column j of P equals M times column j of G_x (= syndrome of unit e_j)
    j = 1234
    e = np.zeros(pp.Gx.N, np.uint32)
    e[j] = 1
    gcol = pp.Gx.syndrome(e)
    assert np.array_equal(pp.PT[j], oracle.server_mvm(pp.W, gcol))


def test_completeness_round_trip(tiny_pp):
    """decode(server(encode(x))) = M x and honest outputs are accepted
    (Def. 4.2 completeness; Thm 6.1 proof)."""
    pp = tiny_pp
    rng = np.random.default_rng(1)
    x_int = rng.integers(-127, 128, pp.n)
    x = oracle.lift(x_int)
    for b in range(3):
        xhat, supp, vals = pp.encrypt(x, oracle.key_from_seed(42), b)
        assert len(supp) == pp.t_x == 163
        assert not np.array_equal(xhat, x)
        yhat = oracle.server_mvm(pp.W, xhat)
        assert pp.verify(xhat, yhat, oracle.key_from_seed(77 + b))
        y = pp.decrypt(supp, vals, yhat)
        assert np.array_equal(oracle.centered(y), pp.W.astype(np.int64) @ x_int)


def test_decrypt_error_identity(tiny_pp):
    """y - Mx = y_hat - M x_hat (soundness proof of Thm 6.1)."""
    pp = tiny_pp
    rng = np.random.default_rng(2)
    x = rng.integers(0, Q, pp.n).astype(np.uint32)
    xhat, supp, vals = pp.encrypt(x, 5, 0)
    yhat = oracle.server_mvm(pp.W, xhat)
    delta = np.zeros(pp.m, np.uint64)
    delta[[3, 100]] = [1, Q - 5]
    y = pp.decrypt(supp, vals, (yhat + delta) % Q)
    assert np.array_equal((y.astype(np.uint64) + Q - oracle.server_mvm(pp.W, x)) % Q, delta)


def test_tampered_outputs_rejected(tiny_pp):
    """With t_y = 31, ell = 2 the acceptance bound is <= 2^-59.9, so every
    tampered output in the sample must be rejected."""
    pp = tiny_pp
    rng = np.random.default_rng(3)
    x = rng.integers(0, Q, pp.n).astype(np.uint32)
    xhat, _, _ = pp.encrypt(x, 6, 0)
    yhat = oracle.server_mvm(pp.W, xhat)
    for trial in range(300):
        bad = yhat.astype(np.uint64).copy()
        kind = trial % 3
        if kind == 0:  # one entry plus a random nonzero constant
            i = rng.integers(pp.m)
            bad[i] = (bad[i] + rng.integers(1, Q)) % Q
        elif kind == 1:  # random dense error
            bad = (bad + rng.integers(0, Q, pp.m)) % Q
        else:  # one wrong row of W
            i = rng.integers(pp.m)
            w2 = pp.W[i].astype(np.int64).copy()
            w2[rng.integers(pp.n)] += 1
            bad[i] = int(np.dot(w2, xhat.astype(object))) % Q
        if np.array_equal(bad, yhat):
            continue
        assert not pp.verify(xhat, bad.astype(np.uint32), oracle.key_from_seed(1000 + trial))


@pytest.mark.parametrize("t", [1, 2, 4])
def test_soundness_rate_matches_lemma_5_1(t):
    """With a weak challenge (t small, ell = 1) the empirical acceptance rate
    of a fixed wrong output matches Pr[supp(e) misses supp(G^T Delta)] =
    C(N - w, t)/C(N, t) (Lemma 5.1; the Schwartz-Zippel term is < 1e-9 here)."""
    rng = np.random.default_rng(t)
    m, n = 4, 6
    W = rng.integers(-127, 128, (m, n)).astype(np.int8)
    pp = oracle.PublicParams(W, oracle.key_from_seed(31), t_x=5, t_y=t, ell=1)
    x = rng.integers(0, Q, n).astype(np.uint32)
    xhat, _, _ = pp.encrypt(x, 8, 0)
    yhat = oracle.server_mvm(W, xhat)
    delta = np.zeros(m, np.uint64)
    delta[1] = 12345
    bad = ((yhat + delta) % Q).astype(np.uint32)
    w = int(np.count_nonzero(pp.Gy.encode(delta)))
    p = oracle.hypergeom_miss(pp.Gy.N, w, t)
    trials = 10000
    acc = sum(pp.verify(xhat, bad, oracle.key_from_seed(10 ** 6 + s)) for s in range(trials))
    sigma = math.sqrt(p * (1 - p) / trials)
    assert abs(acc / trials - p) <= 4 * sigma + 1e-9, (acc / trials, p, w)
    # the honest output is always accepted with the same weak parameters
    assert all(pp.verify(xhat, yhat, oracle.key_from_seed(s)) for s in range(50))


def test_masked_vector_looks_uniform(tiny_pp):
    """Privacy rests on dual-LPN (Thm 6.1): parity unpinned.  Only a sanity
    check: masked entries spread over F_q even for x = 0."""
    pp = tiny_pp
    vals = np.concatenate([pp.encrypt(np.zeros(pp.n, np.uint32), 9, b)[0] for b in range(40)])
    hist = np.bincount((vals.astype(np.uint64) * 16 // Q).astype(np.int64), minlength=16)
    exp = len(vals) / 16
    assert ((hist - exp) ** 2 / exp).sum() < 45


def test_verify_noQ_identity_agrees(tiny_pp):
    """v_L through (G_y e)^T M equals v_L through the stored Q (definition of Q)."""
    pp = tiny_pp
    small = oracle.PublicParams(pp.W, oracle.key_from_seed(0), with_tables=False)
    rng = np.random.default_rng(4)
    x = rng.integers(0, Q, pp.n).astype(np.uint32)
    xhat, supp, vals = pp.encrypt(x, 7, 0)
    yhat = oracle.server_mvm(pp.W, xhat)
    bad = yhat.copy()
    bad[5] = (int(bad[5]) + 1) % Q
    for yh in (yhat, bad):
        assert small.verify(xhat, yh, 99) == pp.verify(xhat, yh, 99)
    rows = [0, 9, 255]
    assert np.array_equal(small.decrypt_rows(supp, vals, yhat[rows], rows),
                          pp.decrypt(supp, vals, yhat)[rows])


# --------------------------------------------------------------------------- Protocol 2

def _bv_claims(rng, B, m, n):
    Ws = [rng.integers(-128, 128, size=(m, n), dtype=np.int8) for _ in range(B)]
    xs = [rng.integers(0, Q, n).astype(np.uint32) for _ in range(B)]
    ys = [oracle.server_mvm(Ws[b], xs[b]) for b in range(B)]
    return Ws, xs, ys


def test_bv_tables_match_dense_definitions():
    """Q_b = G^T M_b and Qaux = Qt^T G' equal the products with the dense App. B
    generators built entry by entry (Protocol 2 preprocessing)."""
    rng = np.random.default_rng(3)
    B, m, n = 2, 3, 2
    Ws, _, _ = _bv_claims(rng, B, m, n)
    bp = oracle.BatchParams(Ws, oracle.key_from_seed(4), t=3, t2=3)
    G, G2 = _dense_G(bp.G), _dense_G(bp.G2)                  # m x N, B n x N'
    GT = [list(col) for col in zip(*G)]                       # N x m
    for b in range(B):
        Mb = [[int(v) % Q for v in row] for row in Ws[b]]     # lifted, m x n
        assert np.array_equal(np.array(_mm(GT, Mb), dtype=np.uint32), bp.Qb[b])
    QtT = [[int(v) for v in row] for row in bp.Qt.T]          # N x B n
    assert np.array_equal(np.array(_mm(QtT, G2), dtype=np.uint32), bp.Qaux)


def test_bv_bilinear_identity():
    """e^T Qaux e' = (G' e')^T (Qt e) for arbitrary e, e' (the identity the
    secondary check relies on), with the syndrome computed independently."""
    rng = np.random.default_rng(5)
    Ws, _, _ = _bv_claims(rng, 3, 4, 3)
    bp = oracle.BatchParams(Ws, oracle.key_from_seed(6), t=5, t2=5)
    for _ in range(5):
        e = rng.integers(0, Q, bp.N).astype(np.uint32)
        e2 = rng.integers(0, Q, bp.N2).astype(np.uint32)
        lhs = sum(int(e[i]) * oracle._dot(bp.Qaux[i], e2) for i in range(bp.N)) % Q
        u = [oracle._dot(bp.Qt[p], e) for p in range(bp.B * bp.n)]
        assert lhs == oracle._dot(bp.G2.syndrome(e2), u)


def test_bv_completeness():
    """Honest outputs and an honest server projection are always accepted."""
    rng = np.random.default_rng(7)
    Ws, xs, ys = _bv_claims(rng, 4, 6, 5)
    bp = oracle.BatchParams(Ws, oracle.key_from_seed(8))
    for s in range(6):
        ch = bp.challenges(oracle.key_from_seed(100 + s))
        assert bp.check(xs, ys, ch, bp.server_project(ch), oracle.key_from_seed(200 + s))


def test_bv_rejects_wrong_outputs_and_projections():
    """A wrong entry in any y_b fails an original check; a server projection
    off by a nonzero vector fails a secondary check (paper parameters)."""
    rng = np.random.default_rng(9)
    Ws, xs, ys = _bv_claims(rng, 3, 5, 4)
    bp = oracle.BatchParams(Ws, oracle.key_from_seed(10))
    for s in range(6):
        ch = bp.challenges(oracle.key_from_seed(300 + s))
        us = bp.server_project(ch)
        bad = [y.copy() for y in ys]
        b, i = s % 3, (2 * s) % 5
        bad[b][i] = (int(bad[b][i]) + 1 + s) % Q
        assert not bp.check(xs, bad, ch, us, oracle.key_from_seed(400 + s))
        ub = us.copy()
        ub[s % bp.ell, (3 * s) % (bp.B * bp.n)] ^= 1
        assert not bp.check(xs, ys, ch, ub, oracle.key_from_seed(500 + s))


@pytest.mark.parametrize("t2", [1, 3])
def test_bv_secondary_rate_matches_lemma_5_1(t2):
    """With a weak secondary challenge (t' small, ell' = 1) a fixed wrong
    projection u = Qt e + Gamma is accepted at the rate
    C(N' - w, t')/C(N', t'), w = wt(G'^T Gamma) (Lemma 5.1 applied to G')."""
    rng = np.random.default_rng(11 + t2)
    Ws, xs, ys = _bv_claims(rng, 2, 3, 3)
    bp = oracle.BatchParams(Ws, oracle.key_from_seed(12), t=4, ell=1, t2=t2, ell2=1)
    ch = bp.challenges(oracle.key_from_seed(13))
    us = bp.server_project(ch)
    gamma = np.zeros(bp.B * bp.n, np.uint64)
    gamma[2] = 777
    bad = ((us + gamma[None, :]) % Q).astype(np.uint32)
    w = int(np.count_nonzero(bp.G2.encode(gamma.astype(np.uint32))))
    p = oracle.hypergeom_miss(bp.N2, w, t2)
    trials = 3000
    acc = sum(bp.check(xs, ys, ch, bad, oracle.key_from_seed(10 ** 6 + s)) for s in range(trials))
    sigma = math.sqrt(p * (1 - p) / trials)
    assert abs(acc / trials - p) <= 4 * sigma + 1e-9, (acc / trials, p, w)
