"""GPU parity: the CUDA path, called through the C-ABI, against the oracle on
the same seeded inputs.  Integer (field) results must match bit for bit."""
import numpy as np
import pytest

import oracle
from gpu_util import (Q, assert_equal_report, ctx_tables, exact_product, field, pt_columns, q_columns,
                      sample_rows, tamper,
                      to_dev)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pv():
    import torch
    assert torch.cuda.is_available()
    import paper_2609_10264_gb300 as pv
    return pv


@pytest.fixture(scope="module")
def wl():
    from paper_2609_10264_gb300 import workloads
    return workloads


def _params(pv, **kw):
    p = pv.pvmvmd_params()
    for k, v in kw.items():
        setattr(p, k, v)
    return p


def _full_round_trip(pv, W, x_int, seeds=(11, 12, 13), params=None, oracle_kw=None):
    """Run preprocess/encode/server/decode_verify on the GPU and the oracle with
    full tables; compare every intermediate exactly."""
    import torch
    m, K = W.shape
    B = x_int.shape[0]
    X = field(x_int)
    Wd = to_dev(W)
    ctx = pv.pvmvmd_preprocess(Wd, key=seeds[0], params=params)
    pp = oracle.PublicParams(W, oracle.key_from_seed(seeds[0]), **(oracle_kw or {}))
    # public codes and tables
    v, tabs = ctx_tables(pv, ctx)
    assert (v.t_x, v.t_y, v.ell) == (pp.t_x, pp.t_y, pp.ell)
    for which, code in (("gx", pp.Gx), ("gy", pp.Gy)):
        for f in ("pi1", "pi2", "v1", "v2"):
            assert np.array_equal(tabs[f"{which}_{f}"], getattr(code, f)), f"{which}_{f}"
    PT = pv.as_u32(pv.device_view(v.PT, v.N_x * m).view(v.N_x, m))
    Qm = pv.as_u32(pv.device_view(v.Q, v.N_y * K).view(v.N_y, K))
    assert np.array_equal(PT, pp.PT)
    assert np.array_equal(Qm, pp.Q)
    # encode
    Xd = to_dev(X)
    Xh, st = pv.pvmvmd_encode(ctx, Xd, key=seeds[1])
    Xh_h, st_h = pv.as_u32(Xh), pv.as_u32(st)
    for b in range(B):
        xh_o, s_o, v_o = pp.encrypt(X[b], oracle.key_from_seed(seeds[1]), b)
        assert np.array_equal(Xh_h[b], xh_o), f"x_hat {b}"
        assert np.array_equal(st_h[b], np.concatenate([s_o, v_o])), f"st {b}"
    # server: batch 1 per vector and the batched call
    Yh1 = torch.stack([pv.pvmvmd_server_mvm(Wd, Xh[b]) for b in range(B)])
    YhB = pv.pvmvmd_server_mvm(Wd, Xh)
    Yh_o = np.stack([oracle.server_mvm(W, Xh_h[b]) for b in range(B)])
    assert np.array_equal(pv.as_u32(Yh1), Yh_o)
    assert np.array_equal(pv.as_u32(YhB), Yh_o)
    # decode + verify
    Y, acc = pv.pvmvmd_decode_verify(ctx, st, Xh, YhB, challenge_key=seeds[2])
    Y_h = pv.as_u32(Y)
    for b in range(B):
        assert np.array_equal(Y_h[b], pp.decrypt(st_h[b, :pp.t_x], st_h[b, pp.t_x:], Yh_o[b]))
        assert np.array_equal(oracle.centered(Y_h[b]), W.astype(np.int64) @ x_int[b])
    assert pv.as_u32(acc).tolist() == [1] * B
    assert all(pp.verify(Xh_h[b], Yh_o[b], oracle.key_from_seed(seeds[2])) for b in range(B))
    # tampered outputs: rejected by both
    bad = YhB.clone()
    rng = np.random.default_rng(0)
    for b in range(0, B, 2):
        tamper(pv, bad, b, int(rng.integers(m)), int(rng.integers(1, Q)))
    bad_h = pv.as_u32(bad)
    _, acc_bad = pv.pvmvmd_decode_verify(ctx, st, Xh, bad, challenge_key=seeds[2] + 1)
    exp = [0 if b % 2 == 0 else 1 for b in range(B)]
    assert pv.as_u32(acc_bad).tolist() == exp
    for b in range(0, B, 2):
        assert not pp.verify(Xh_h[b], bad_h[b], oracle.key_from_seed(seeds[2] + 1))
    # in place: Y overwrites Y_hat, so the check reads Y_hat before the decrypt
    Yip = YhB.clone()
    _, acc_ip = pv.pvmvmd_decode_verify(ctx, st, Xh, Yip, challenge_key=seeds[2], Y=Yip)
    assert np.array_equal(pv.as_u32(Yip), Y_h)
    assert pv.as_u32(acc_ip).tolist() == [1] * B
    bad_ip = bad.clone()
    _, acc_bad_ip = pv.pvmvmd_decode_verify(ctx, st, Xh, bad_ip, challenge_key=seeds[2] + 1, Y=bad_ip)
    assert pv.as_u32(acc_bad_ip).tolist() == exp
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()


def test_config1_tiny_round_trip(pv, wl):
    """256 x 256 uniform int8 weights, one int8 vector from seed 0 (config 1)."""
    W = wl.weights_uniform(256, 256, 0)
    x = wl.int8_vectors(1, 256, 0)
    _full_round_trip(pv, W, x, seeds=(0, 0, 0))


@pytest.mark.parametrize("m,K,B", [(37, 100, 3), (300, 1000, 5), (129, 48, 2), (4, 40, 1), (513, 33, 4)])
def test_ragged_round_trip(pv, wl, m, K, B):
    W = wl.weights_uniform(m, K, m * 7 + K)
    x = wl.int8_vectors(B, K, m + K)
    _full_round_trip(pv, W, x, seeds=(m, K, B))


def test_small_parameters_round_trip(pv, wl):
    """Non-default rate and sparsities (rate 3, t_x 5, t_y 3, ell 3)."""
    W = wl.weights_uniform(20, 12, 5)
    x = wl.int8_vectors(3, 12, 6)
    params = _params(pv, rate=3, t_x=5, t_y=3, ell=3)
    _full_round_trip(pv, W, x, seeds=(3, 4, 5), params=params,
                     oracle_kw=dict(t_x=5, t_y=3, ell=3, rate=3))


def test_encode_chunking_matches(pv, wl):
    """Encoding in chunks of 3 vectors (scratch_batch) gives the same result."""
    W = wl.weights_uniform(64, 96, 1)
    X = field(wl.int8_vectors(8, 96, 2))
    Wd, Xd = to_dev(W), to_dev(X)
    a = pv.pvmvmd_preprocess(Wd, key=9)
    b = pv.pvmvmd_preprocess(Wd, key=9, params=_params(pv, scratch_batch=3))
    xa, sa = pv.pvmvmd_encode(a, Xd, key=10)
    xb, sb = pv.pvmvmd_encode(b, Xd, key=10)
    assert np.array_equal(pv.as_u32(xa), pv.as_u32(xb))
    assert np.array_equal(pv.as_u32(sa), pv.as_u32(sb))
    # in place (X and Xhat alias)
    xc = Xd.clone()
    pv.pvmvmd_encode(a, xc, key=10, Xhat=xc)
    assert np.array_equal(pv.as_u32(xc), pv.as_u32(xa))


def test_lane_encode_ragged_groups_and_chunks(pv, wl):
    """Batches large enough for the lane-parallel encode, on a code too long for
    one CTA (K = 6000, N_x = 48000): 300 vectors in chunks of 270 (two lane
    groups of 256 and 14 lanes, then a 30-lane chunk) and a ragged 33-vector
    batch; every x_hat and mask equals the oracle, and the chunked and
    unchunked contexts agree."""
    W = wl.weights_uniform(40, 6000, 21)
    x = wl.int8_vectors(300, 6000, 22)
    X = field(x)
    Wd, Xd = to_dev(W), to_dev(X)
    pp = oracle.PublicParams(W, oracle.key_from_seed(23), with_tables=False)
    a = pv.pvmvmd_preprocess(Wd, key=23, params=_params(pv, scratch_batch=270))
    b = pv.pvmvmd_preprocess(Wd, key=23, params=_params(pv, scratch_batch=300))
    xa, sa = pv.pvmvmd_encode(a, Xd, key=24)
    xb, sb = pv.pvmvmd_encode(b, Xd, key=24)
    xa_h, sa_h = pv.as_u32(xa), pv.as_u32(sa)
    for i in range(300):
        xh_o, s_o, v_o = pp.encrypt(X[i], oracle.key_from_seed(24), i)
        assert np.array_equal(xa_h[i], xh_o), i
        assert np.array_equal(sa_h[i], np.concatenate([s_o, v_o])), i
    assert np.array_equal(pv.as_u32(xb), xa_h)
    assert np.array_equal(pv.as_u32(sb), sa_h)
    # 33 vectors (one lane group, a ragged warp), in place
    xc = Xd[:33].clone()
    pv.pvmvmd_encode(a, xc, key=24, Xhat=xc)
    assert np.array_equal(pv.as_u32(xc), xa_h[:33])
    assert pv.pvmvmd_device_status() == 0
    a.destroy()
    b.destroy()


@pytest.mark.parametrize("m,K,B", [(300, 1000, 5), (64, 6000, 40), (4096, 4096, 3)])
def test_boost_mode_matches_standard_mode(pv, wl, m, K, B):
    """Boost mode (masks prepared ahead) gives the same x_hat, y and verdicts
    as the standard calls with the same keys; the masks equal the oracle's
    G_x e_x and P e_x; a tampered output is rejected."""
    W = wl.weights_uniform(m, K, m + K)
    x = wl.int8_vectors(B, K, m + 2 * K)
    X = field(x)
    Wd, Xd = to_dev(W), to_dev(X)
    ctx = pv.pvmvmd_preprocess(Wd, key=41)
    pp = oracle.PublicParams(W, oracle.key_from_seed(41), with_tables=False)
    mi, mo, st = pv.pvmvmd_boost_prepare(ctx, B, key=42)
    mi_h, mo_h, st_h = pv.as_u32(mi), pv.as_u32(mo), pv.as_u32(st)
    zeros = np.zeros(K, np.uint32)
    for b in range(B):
        xp, s_o, v_o = pp.encrypt(zeros, oracle.key_from_seed(42), b)
        assert np.array_equal(mi_h[b], xp), b
        assert np.array_equal(st_h[b], np.concatenate([s_o, v_o])), b
        rows = sample_rows(m, 16, b)
        y0 = np.zeros(len(rows), np.uint32)
        neg = pp.decrypt_rows(s_o, v_o, y0, rows)  # 0 - P e_x on the sampled rows
        assert np.array_equal((Q - neg.astype(np.int64)) % Q, mo_h[b, rows].astype(np.int64)), b
    Xh = pv.pvmvmd_boost_encode(Xd, mi)
    Xs, sts = pv.pvmvmd_encode(ctx, Xd, key=42)
    assert np.array_equal(pv.as_u32(Xh), pv.as_u32(Xs))
    Yh = pv.pvmvmd_server_mvm(Wd, Xh)
    Yb, ab = pv.pvmvmd_boost_decode_verify(ctx, mo, Xh, Yh, challenge_key=43)
    Ys, as_ = pv.pvmvmd_decode_verify(ctx, sts, Xs, Yh, challenge_key=43)
    assert np.array_equal(pv.as_u32(Yb), pv.as_u32(Ys))
    assert np.array_equal(oracle.centered(pv.as_u32(Yb)), x.astype(np.int64) @ W.astype(np.int64).T)
    assert pv.as_u32(ab).tolist() == [1] * B and pv.as_u32(as_).tolist() == [1] * B
    tamper(pv, Yh, B - 1, m // 2, 7)
    _, ab2 = pv.pvmvmd_boost_decode_verify(ctx, mo, Xh, Yh, challenge_key=44)
    assert pv.as_u32(ab2).tolist() == [1] * (B - 1) + [0]
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()


@pytest.mark.parametrize("B,m,n", [(3, 40, 30), (4, 96, 64), (2, 700, 600)])
def test_batch_verification_protocol2(pv, wl, B, m, n):
    """Protocol 2 on the GPU against the oracle: the preprocessed Qs and
    Qaux, the server projection, the secondary challenges, and the verdicts
    on honest claims, a wrong output and a wrong projection."""
    import torch
    rng = np.random.default_rng(B * 1000 + m + n)
    Ws = rng.integers(-128, 128, size=(B, m, n), dtype=np.int8)
    xs = rng.integers(0, Q, size=(B, n)).astype(np.uint32)
    ys = np.stack([oracle.server_mvm(Ws[b], xs[b]) for b in range(B)])
    ctx = pv.pvmvmd_bv_preprocess(to_dev(Ws), key=51)
    bp = oracle.BatchParams(list(Ws), oracle.key_from_seed(51))
    assert (ctx.N, ctx.N2, ctx.t, ctx.ell, ctx.t2, ctx.ell2) == (bp.N, bp.N2, bp.t, bp.ell, bp.t2, bp.ell2)
    Qs = pv.as_u32(pv.device_view(ctx.Qs, ctx.N * B * n).view(ctx.N, B * n))
    assert np.array_equal(Qs, bp.Qt.T)
    cols = sample_rows(ctx.N2, 16, 3)
    QauxT = pv.device_view(ctx.QauxT, ctx.N2 * ctx.N).view(ctx.N2, ctx.N)
    assert np.array_equal(pv.as_u32(QauxT[torch.as_tensor(cols, device=QauxT.device)]), bp.Qaux[:, cols].T)
    chal = pv.pvmvmd_bv_challenge(ctx, key=52)
    ch_o = bp.challenges(oracle.key_from_seed(52))
    ch_h = pv.as_u32(chal)
    for q, (s_o, v_o) in enumerate(ch_o):
        assert np.array_equal(ch_h[q], np.concatenate([s_o, v_o]))
    u = pv.pvmvmd_bv_server_project(ctx, chal)
    assert np.array_equal(pv.as_u32(u), bp.server_project(ch_o))
    Xd, Yd = to_dev(xs), to_dev(ys)
    acc = pv.pvmvmd_bv_check(ctx, Xd, Yd, chal, u, key2=53)
    assert pv.as_u32(acc).tolist() == [1]
    assert bp.check(list(xs), list(ys), ch_o, bp.server_project(ch_o), oracle.key_from_seed(53))
    sec = pv.as_u32(pv.device_view(ctx.chal2, ctx.ell2 * 2 * ctx.t2).view(ctx.ell2, 2 * ctx.t2))
    for j, (s_o, v_o) in enumerate(bp.secondary(oracle.key_from_seed(53))):
        assert np.array_equal(sec[j], np.concatenate([s_o, v_o]))
    # a wrong output, then a wrong projection: rejected by both
    bad = ys.copy()
    bad[B - 1, m // 3] = (int(bad[B - 1, m // 3]) + 9) % Q
    assert pv.as_u32(pv.pvmvmd_bv_check(ctx, Xd, to_dev(bad), chal, u, key2=54)).tolist() == [0]
    assert not bp.check(list(xs), list(bad), ch_o, bp.server_project(ch_o), oracle.key_from_seed(54))
    ub = u.clone()
    tamper(pv, ub, 0, (B * n) // 2, 3)
    assert pv.as_u32(pv.pvmvmd_bv_check(ctx, Xd, Yd, chal, ub, key2=55)).tolist() == [0]
    assert not bp.check(list(xs), list(ys), ch_o, pv.as_u32(ub), oracle.key_from_seed(55))
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()


@pytest.mark.parametrize("B", [1, 5, 40])
def test_sixteen_bit_weights_round_trip(pv, wl, B):
    """16-bit weights (Sec. 7.2 style, including both ends of the supported
    range): the split planes recombine to M; P^T and Q equal 256 x the
    tables of M_hi plus those of M_lo (linearity, each from the oracle); the
    decrypted output equals the exact integer product W x for every vector."""
    import torch
    rng = np.random.default_rng(70 + B)
    m, K = 300, 1000
    W = rng.integers(-32768, 32640, size=(m, K)).astype(np.int16)
    W[0, :5] = [-32768, 32639, -1, 0, 255]
    x = rng.integers(-8, 9, size=(B, K)).astype(np.int64)       # |W x| < q / 2
    Wd = torch.from_numpy(W).cuda()
    hi, lo = pv.pvmvmd_weights_split_i16(Wd)
    hi_h, lo_h = hi.cpu().numpy(), lo.cpu().numpy()
    assert np.array_equal(256 * hi_h.astype(np.int64) + lo_h.astype(np.int64), W.astype(np.int64))
    ctx = pv.pvmvmd_preprocess_i16(Wd, key=71)
    v = pv.pvmvmd_ctx_info(ctx)
    ph = oracle.PublicParams(hi_h, oracle.key_from_seed(71))
    pl = oracle.PublicParams(lo_h, oracle.key_from_seed(71))
    PT = pv.as_u32(pv.device_view(v.PT, v.N_x * m).view(v.N_x, m)).astype(np.int64)
    Qm = pv.as_u32(pv.device_view(v.Q, v.N_y * K).view(v.N_y, K)).astype(np.int64)
    assert np.array_equal(PT, (256 * ph.PT.astype(np.int64) + pl.PT) % Q)
    assert np.array_equal(Qm, (256 * ph.Q.astype(np.int64) + pl.Q) % Q)
    Xh, st = pv.pvmvmd_encode(ctx, to_dev(field(x)), key=72)
    Yh = pv.pvmvmd_server_mvm_i16(hi, lo, Xh if B > 1 else Xh[0])
    Yh2 = Yh.view(B, m)
    Y, acc = pv.pvmvmd_decode_verify(ctx, st, Xh, Yh2, challenge_key=73)
    assert pv.as_u32(acc).tolist() == [1] * B
    assert np.array_equal(oracle.centered(pv.as_u32(Y)), x @ W.astype(np.int64).T)
    tamper(pv, Yh2, 0, 7, 1)
    _, acc2 = pv.pvmvmd_decode_verify(ctx, st, Xh, Yh2, challenge_key=74)
    assert pv.as_u32(acc2).tolist() == [0] + [1] * (B - 1)
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()


def test_server_mvm_extremes(pv):
    """Extreme weights and field values: -128, 127, x = 0, 1, (q-1)/2, (q+1)/2, q-1."""
    rng = np.random.default_rng(1)
    for m, K in ((64, 4096), (17, 1000), (8, 16)):
        W = rng.choice(np.array([-128, -127, 127, 0, 1], np.int8), size=(m, K))
        W[0] = -128
        W[1] = 127
        vals = np.array([0, 1, (Q - 1) // 2, (Q + 1) // 2, Q - 1, Q - 2], np.uint32)
        X = rng.choice(vals, size=(3, K)).astype(np.uint32)
        X[0] = Q - 1
        X[1] = (Q + 1) // 2
        Wd = to_dev(W)
        Xd = to_dev(X)
        exp = np.stack([oracle.server_mvm(W, X[b]) for b in range(3)])
        assert np.array_equal(pv.as_u32(pv.pvmvmd_server_mvm(Wd, Xd)), exp)
        assert np.array_equal(pv.as_u32(pv.pvmvmd_server_mvm(Wd, Xd[0])), exp[0])


@pytest.mark.parametrize("B", [1, 8, 64])
@pytest.mark.parametrize("K", [131071, 131056])
def test_server_mvm_max_k(pv, K, B):
    """The largest K the ABI accepts (and the largest multiple of 16 below
    it) on each server path, at the digit sums' extreme: M = -128 against
    x_hat centred at -128 (1 + 2^8 + 2^16), whose three low signed base-256
    digits are all -128, so each of those exact digit sums is 16384 K, just
    below 2^31."""
    assert K <= pv.PVMVMD_MAX_K and 16384 * pv.PVMVMD_MAX_K < 2**31
    rng = np.random.default_rng(K + B)
    W = rng.integers(-128, 128, size=(5, K), dtype=np.int8)
    W[0] = -128
    W[1] = 127
    low = 128 * (1 + 256 + 65536)
    X = rng.integers(0, Q, size=(B, K)).astype(np.uint32)
    X[0] = Q - low                 # centred -low: digits (-128, -128, -128, 0)
    if B > 1:
        X[1] = (1 << 24) - low     # digits (-128, -128, -128, 1)
    got = pv.as_u32(pv.pvmvmd_server_mvm(to_dev(W), to_dev(X if B > 1 else X[0])))
    exp = np.stack([oracle.server_mvm(W, X[b]) for b in range(B)])
    assert np.array_equal(got.reshape(B, 5), exp)
    assert pv.pvmvmd_device_status() == 0


def test_server_mvm_long_k_segments(pv):
    """K beyond one shared-memory segment of digit planes (60000 > 49152)."""
    rng = np.random.default_rng(2)
    W = rng.integers(-128, 128, size=(40, 60000), dtype=np.int8)
    x = rng.integers(0, Q, 60000).astype(np.uint32)
    got = pv.as_u32(pv.pvmvmd_server_mvm(to_dev(W), to_dev(x)))
    assert np.array_equal(got, oracle.server_mvm(W, x))


def test_config2_gemv_all_vectors(pv, wl):
    """4096 x 4096 Gaussian(32) int8 weights, 100 vectors uniform in F_q, batch 1."""
    import torch
    W = wl.weights_gaussian(4096, 4096, 2)
    X = wl.field_vectors(100, 4096, 2)
    Wd, Xd = to_dev(W), to_dev(X)
    got = torch.stack([pv.pvmvmd_server_mvm(Wd, Xd[b]) for b in range(100)])
    got = pv.as_u32(got)
    for b in range(100):
        assert np.array_equal(got[b], oracle.server_mvm(W, X[b])), b


def test_config2_round_trip(pv, wl):
    """Full pipeline at 4096 x 4096 with 100 int8 vectors; tables compared in full."""
    import torch
    W = wl.weights_gaussian(4096, 4096, 2)
    x = wl.int8_vectors(100, 4096, 3)
    X = field(x)
    Wd = to_dev(W)
    ctx = pv.pvmvmd_preprocess(Wd, key=20)
    pp = oracle.PublicParams(W, oracle.key_from_seed(20))
    v = pv.pvmvmd_ctx_info(ctx)
    assert np.array_equal(pv.as_u32(pv.device_view(v.PT, v.N_x * 4096).view(v.N_x, 4096)), pp.PT)
    assert np.array_equal(pv.as_u32(pv.device_view(v.Q, v.N_y * 4096).view(v.N_y, 4096)), pp.Q)
    Xh, st = pv.pvmvmd_encode(ctx, to_dev(X), key=21)
    Yh = torch.stack([pv.pvmvmd_server_mvm(Wd, Xh[b]) for b in range(100)])
    Y, acc = pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, challenge_key=22)
    Xh_h, st_h, Yh_h, Y_h = pv.as_u32(Xh), pv.as_u32(st), pv.as_u32(Yh), pv.as_u32(Y)
    for b in range(100):
        xh_o, s_o, v_o = pp.encrypt(X[b], oracle.key_from_seed(21), b)
        assert np.array_equal(Xh_h[b], xh_o)
        assert np.array_equal(st_h[b], np.concatenate([s_o, v_o]))
        assert np.array_equal(Yh_h[b], oracle.server_mvm(W, xh_o))
        assert np.array_equal(Y_h[b], pp.decrypt(s_o, v_o, Yh_h[b]))
    # every partial sum is below 2^53, so the float64 product is exact
    assert np.array_equal(oracle.centered(Y_h), (x.astype(np.float64) @ W.astype(np.float64).T).astype(np.int64))
    assert pv.as_u32(acc).tolist() == [1] * 100
    for b in (0, 57, 99):
        assert pp.verify(Xh_h[b], Yh_h[b], oracle.key_from_seed(22))
    tamper(pv, Yh, 3, 5, 1)
    tamper(pv, Yh, 50, 4095, Q - 1)
    _, acc2 = pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, challenge_key=23)
    a2 = pv.as_u32(acc2)
    assert a2[3] == 0 and a2[50] == 0 and a2.sum() == 98
    assert pv.pvmvmd_device_status() == 0


@pytest.mark.parametrize("layer", [0, 31])
def test_config3_layer_gemv(pv, wl, layer):
    """One 8B-class decoder layer at batch 1 (7 projections), every output."""
    for j, (name, (m, K)) in enumerate(wl.LAYER_8B.items()):
        W = wl.weights_gaussian(m, K, (3, layer, j))
        x = wl.field_vectors(1, K, (3, layer, j, 1))[0]
        got = pv.as_u32(pv.pvmvmd_server_mvm(to_dev(W), to_dev(x)))
        assert_equal_report(got, oracle.server_mvm_batch(W, x)[0], name)


def _batched_pipeline(pv, W, B, seed, n_rows=24, n_verify=2):
    """Preprocess/encode/server/decode_verify at a large shape.  Checks: P^T
    and Q columns, every x_hat and mask, every element of the server's output
    against the oracle, every decoded element against the exact integer
    product (completeness), all accepted, and the oracle's verdict and
    decryption for a few vectors."""
    m, K = W.shape
    x = np.random.default_rng(seed).integers(-127, 128, size=(B, K), dtype=np.int64)
    X = field(x)
    Wd = to_dev(W)
    ctx = pv.pvmvmd_preprocess(Wd, key=seed)
    pp = oracle.PublicParams(W, oracle.key_from_seed(seed), with_tables=False)
    rows = sample_rows(m, n_rows, seed)
    cols = sample_rows(K, n_rows, seed + 1)
    ptc = pt_columns(pv, ctx, rows)
    for i, r in enumerate(rows):
        assert np.array_equal(ptc[:, i], pp.Gx.encode(oracle.lift(W[r]))), f"P^T column {r}"
    qc = q_columns(pv, ctx, cols)
    for i, c in enumerate(cols):
        assert np.array_equal(qc[:, i], pp.Gy.encode(oracle.lift(W[:, c]))), f"Q column {c}"
    Xh, st = pv.pvmvmd_encode(ctx, to_dev(X), key=seed + 1)
    Xh_h, st_h = pv.as_u32(Xh), pv.as_u32(st)
    for b in range(B):
        xh_o, s_o, v_o = pp.encrypt(X[b], oracle.key_from_seed(seed + 1), b)
        assert np.array_equal(Xh_h[b], xh_o), b
        assert np.array_equal(st_h[b], np.concatenate([s_o, v_o])), b
    Yh = pv.pvmvmd_server_mvm(Wd, Xh)
    Yh_h = pv.as_u32(Yh)
    # every output element, bit for bit
    assert_equal_report(Yh_h, oracle.server_mvm_batch(W, Xh_h), "server product")
    Y, acc = pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, challenge_key=seed + 2)
    Y_h = pv.as_u32(Y)
    # completeness on every element: y = W x exactly (|W x| < q / 2)
    assert_equal_report(oracle.centered(Y_h), exact_product(W, x), "decrypted output")
    assert pv.as_u32(acc).tolist() == [1] * B
    for b in range(n_verify):
        assert pp.verify(Xh_h[b], Yh_h[b], oracle.key_from_seed(seed + 2))
        assert np.array_equal(Y_h[b, rows[:4]], pp.decrypt_rows(st_h[b, :pp.t_x], st_h[b, pp.t_x:],
                                                                 Yh_h[b, rows[:4]], rows[:4]))
    tamper(pv, Yh, 1, int(rows[1]), 1)
    _, acc2 = pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, challenge_key=seed + 3)
    a2 = pv.as_u32(acc2)
    assert a2[1] == 0 and a2.sum() == B - 1
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()


@pytest.mark.parametrize("name", ["q", "k", "gate", "down"])
def test_config4_batched_8b(pv, wl, name):
    """8B-class layer shapes with 64 vectors per call (the batched product)."""
    m, K = wl.LAYER_8B[name]
    W = wl.weights_gaussian(m, K, (4, list(wl.LAYER_8B).index(name)))
    _batched_pipeline(pv, W, 64, seed=400 + len(name))


@pytest.mark.parametrize("name", ["q", "kv", "gate_up", "down"])
def test_config5_70b(pv, wl, name):
    """70B-class shapes with 256 vectors per call; the largest K is 28672."""
    m, K = wl.LAYER_70B[name]
    W = wl.weights_gaussian(m, K, (5, list(wl.LAYER_70B).index(name)))
    _batched_pipeline(pv, W, 256, seed=500 + len(name), n_rows=12, n_verify=1)


@pytest.mark.parametrize("m,K,B", [
    (600, 1000, 70),      # K % 16 != 0: byte-load path; two vector tiles, the second ragged
    (513, 4144, 130),     # TMA path; m crosses a CTA pair by one row; K % 64 = 48; three vector tiles
    (1030, 16384, 257),   # five row pairs (the last ragged), five vector tiles (one vector in the last)
    (257, 4100, 65),      # byte-load path, ragged in every dimension
    (4096, 4096, 64),     # an 8B-class projection with 64 vectors (K split over the cluster)
    (128, 8192, 512),     # one CTA pair on half-used rows, eight vector tiles, long K
])
def test_batched_product_full_multi_tile(pv, m, K, B):
    """The tensor-core product on shapes that span several CTA pairs, vector
    tiles and K-split ranks with ragged edges in m, K and B: every output
    element equals the oracle's, with extreme weights and x_hat in some rows
    and vectors."""
    rng = np.random.default_rng(m * 7 + K * 3 + B)
    W = rng.integers(-128, 128, size=(m, K), dtype=np.int8)
    W[0] = -128
    W[m - 1] = 127
    X = rng.integers(0, Q, size=(B, K)).astype(np.uint32)
    X[0] = (Q + 1) // 2
    X[B - 1] = Q - 1
    Y = pv.as_u32(pv.pvmvmd_server_mvm(to_dev(W), to_dev(X)))
    assert_equal_report(Y, oracle.server_mvm_batch(W, X), f"{m}x{K}x{B}")
    assert pv.pvmvmd_device_status() == 0


def test_server_mvm_concurrent_streams(pv, wl):
    """Batched and small-batch products issued on two streams at once keep
    their digit operands apart: every output equals the oracle's."""
    import torch
    cases = [(512, 3072, 64), (384, 2048, 96), (700, 1024, 8), (256, 4096, 12)]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    ins, outs = [], []
    for j, (m, K, B) in enumerate(cases):
        W = wl.weights_uniform(m, K, (51, j))
        X = np.random.default_rng(52 + j).integers(0, Q, size=(B, K), dtype=np.int64).astype(np.uint32)
        ins.append((W, X, to_dev(W), to_dev(X)))
    torch.cuda.synchronize()
    for rep in range(3):
        outs = []
        for j, (W, X, Wd, Xd) in enumerate(ins):
            s = streams[j % 2]
            with torch.cuda.stream(s):
                outs.append(pv.pvmvmd_server_mvm(Wd, Xd, stream=s))
        torch.cuda.synchronize()
    for (W, X, _, _), Yh in zip(ins, outs):
        assert_equal_report(pv.as_u32(Yh), oracle.server_mvm_batch(W, X), str(W.shape))
    assert pv.pvmvmd_device_status() == 0


@pytest.mark.parametrize("L", [256, 128])
def test_lane_encode_long_tiles(pv, wl, L):
    """The lane encode on a long code (K = 28672, N_x = 229376) with every
    vector in one lane group: on a 152-SM GB300, 256 lanes run the tile sums
    and the scan over tiles of 128 positions, 128 lanes over tiles of 64;
    every x_hat and state equals the oracle."""
    W = wl.weights_uniform(24, 28672, 31)
    x = wl.int8_vectors(L, 28672, 32)
    X = field(x)
    ctx = pv.pvmvmd_preprocess(to_dev(W), key=33, params=_params(pv, scratch_batch=L))
    pp = oracle.PublicParams(W, oracle.key_from_seed(33), with_tables=False)
    Xh, st = pv.pvmvmd_encode(ctx, to_dev(X), key=34)
    Xh_h, st_h = pv.as_u32(Xh), pv.as_u32(st)
    for b in range(L):
        xh_o, s_o, v_o = pp.encrypt(X[b], oracle.key_from_seed(34), b)
        assert np.array_equal(Xh_h[b], xh_o), b
        assert np.array_equal(st_h[b], np.concatenate([s_o, v_o])), b
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()


@pytest.mark.parametrize("m,K,B", [(4096, 2560, 8), (37, 6144 + 96, 5), (300, 16, 2), (2560, 9728, 16),
                                   (1000, 4096, 3)])
def test_small_batch_server_product(pv, wl, m, K, B):
    """2 <= B <= 16 runs the small-batch GEMV (one pass over M per four
    vectors, K in segments of 6144): equal to the per-vector GEMV and to the
    oracle on every output, with full-range x_hat and extreme weights."""
    import torch
    rng = np.random.default_rng(m + K + B)
    W = rng.integers(-128, 128, size=(m, K), dtype=np.int8)
    W[0, :] = -128
    X = rng.integers(0, Q, size=(B, K)).astype(np.uint32)
    X[0, :] = (Q - 1) // 2 + 1
    Wd, Xd = to_dev(W), to_dev(X)
    Y = pv.as_u32(pv.pvmvmd_server_mvm(Wd, Xd))
    Y1 = np.stack([pv.as_u32(pv.pvmvmd_server_mvm(Wd, Xd[b])) for b in range(B)])
    assert np.array_equal(Y, Y1)
    assert_equal_report(Y, oracle.server_mvm_batch(W, X), "small-batch product")
    assert pv.pvmvmd_device_status() == 0


@pytest.mark.parametrize("name", ["q", "o", "down"])
def test_qwen3_4b_block_8_tokens(pv, wl, name):
    """Qwen3-4B projection shapes (the paper's evaluation table) with an
    eight-token batch, synthetic weights."""
    m, K = wl.LAYER_QWEN3_4B[name]
    W = wl.weights_gaussian(m, K, (6, list(wl.LAYER_QWEN3_4B).index(name)))
    _batched_pipeline(pv, W, 8, seed=600 + len(name))


def test_server_mvm_multi_mixed_jobs(pv, wl):
    """Grouped batch-1 products over mixed shapes, including K beyond one
    segment (20000), a K that is not a multiple of 16 (1001) and tiny matrices; equal to the
    single calls and to the oracle."""
    import torch
    rng = np.random.default_rng(7)
    shapes = [(4096, 4096), (1024, 4096), (300, 20000), (17, 1001), (5, 16), (64, 48), (2048, 14336)]
    W = [rng.integers(-128, 128, size=s, dtype=np.int8) for s in shapes]
    X = [rng.integers(0, Q, size=s[1]).astype(np.uint32) for s in shapes]
    Wd = [to_dev(w) for w in W]
    Xd = [to_dev(x) for x in X]
    Yd = [torch.empty(s[0], dtype=torch.int32, device="cuda") for s in shapes]
    pv.pvmvmd_server_mvm_multi(list(zip(Wd, Xd, Yd)))
    for i, s in enumerate(shapes):
        single = pv.as_u32(pv.pvmvmd_server_mvm(Wd[i], Xd[i]))
        got = pv.as_u32(Yd[i])
        assert np.array_equal(got, single), s
        assert_equal_report(got, oracle.server_mvm_batch(W[i], X[i])[0], str(s))
    # many jobs (more than one launch's worth) on replicas of one matrix
    Wr = Wd[4]
    Xs = to_dev(rng.integers(0, Q, size=(300, 16)).astype(np.uint32))
    Ys = torch.empty((300, 5), dtype=torch.int32, device="cuda")
    pv.pvmvmd_server_mvm_multi([(Wr, Xs[b], Ys[b]) for b in range(300)])
    Xs_h = pv.as_u32(Xs)
    assert np.array_equal(pv.as_u32(Ys), np.stack([oracle.server_mvm(W[4], Xs_h[b]) for b in range(300)]))
    assert pv.pvmvmd_device_status() == 0


@pytest.mark.parametrize("m,K,B,sb", [(4096, 4096, 8, 0),      # fused encode and challenges
                                       (16, 50000, 3, 0),       # sample / scan / gather encode
                                       (1024, 8192, 40, 40)])   # lane-parallel encode
def test_encode_overlaps_decode(pv, wl, m, K, B, sb):
    """An encode may run on another stream while an earlier batch of the
    same context is decoded: both give exactly what they give in order."""
    import torch
    W = wl.weights_uniform(m, K, 70 + B)
    x1, x2 = wl.int8_vectors(B, K, 71), wl.int8_vectors(B, K, 72)
    params = _params(pv, scratch_batch=sb) if sb else None
    Wd = to_dev(W)
    ctx = pv.pvmvmd_preprocess(Wd, key=73, params=params)
    X1, X2 = to_dev(field(x1)), to_dev(field(x2))
    Xh1, st1 = pv.pvmvmd_encode(ctx, X1, key=74)
    Yh1 = pv.pvmvmd_server_mvm(Wd, Xh1)
    # in order
    Xh2_ref, st2_ref = pv.pvmvmd_encode(ctx, X2, key=75)
    Y1_ref, acc_ref = pv.pvmvmd_decode_verify(ctx, st1, Xh1, Yh1, challenge_key=76)
    torch.cuda.synchronize()
    assert pv.as_u32(acc_ref).tolist() == [1] * B
    assert np.array_equal(oracle.centered(pv.as_u32(Y1_ref)), x1.astype(np.int64) @ W.astype(np.int64).T)
    # overlapped: the decode on one stream, the next batch's encode on another
    sa, sb_ = torch.cuda.Stream(), torch.cuda.Stream()
    Xh2, st2 = torch.empty_like(Xh2_ref), torch.empty_like(st2_ref)
    Y1, acc = torch.empty_like(Y1_ref), torch.empty_like(acc_ref)
    for _ in range(3):
        ev = torch.cuda.Event()
        ev.record(torch.cuda.current_stream())
        sa.wait_event(ev)
        sb_.wait_event(ev)
        Xh2.zero_(); st2.zero_(); Y1.zero_(); acc.zero_()
        ev2 = torch.cuda.Event()
        ev2.record(torch.cuda.current_stream())
        sa.wait_event(ev2)
        sb_.wait_event(ev2)
        pv.pvmvmd_decode_verify(ctx, st1, Xh1, Yh1, challenge_key=76, Y=Y1, accept=acc, stream=sa)
        pv.pvmvmd_encode(ctx, X2, key=75, Xhat=Xh2, st=st2, stream=sb_)
        torch.cuda.synchronize()
        assert np.array_equal(pv.as_u32(Xh2), pv.as_u32(Xh2_ref))
        assert np.array_equal(pv.as_u32(st2), pv.as_u32(st2_ref))
        assert np.array_equal(pv.as_u32(Y1), pv.as_u32(Y1_ref))
        assert pv.as_u32(acc).tolist() == [1] * B
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()


@pytest.mark.parametrize("m,K,which,L", [(64, 300, 0, 300), (300, 64, 1, 257), (4096, 4096, 0, 4096)])
def test_code_encode_lanes(pv, wl, m, K, which, L):
    """G^T over lanes (the encoder of App. B that preprocessing runs) equals
    the oracle's encoding lane by lane, with ragged lane blocks; with the
    rows of M as lanes it reproduces the context's P^T."""
    W = wl.weights_uniform(m, K, 90)
    ctx = pv.pvmvmd_preprocess(to_dev(W), key=91)
    pp = oracle.PublicParams(W, oracle.key_from_seed(91), with_tables=False)
    code = pp.Gx if which == 0 else pp.Gy
    n = K if which == 0 else m
    rng = np.random.default_rng(92)
    X = rng.integers(0, Q, size=(n, L)).astype(np.uint32)
    X[:, 0] = Q - 1
    X[:, -1] = 0
    Y = pv.as_u32(pv.pvmvmd_code_encode_lanes(ctx, which, to_dev(X)))
    assert Y.shape == (n * ctx.rate, L)
    for l in sorted({0, 1, L // 2, L - 1, *rng.integers(0, L, 8).tolist()}):
        assert np.array_equal(Y[:, l], code.encode(X[:, l])), l
    if which == 0 and L == m:
        v, _ = ctx_tables(pv, ctx)
        PT = pv.as_u32(pv.device_view(v.PT, v.N_x * m).view(v.N_x, m))
        got = pv.as_u32(pv.pvmvmd_code_encode_lanes(ctx, 0, to_dev(field(W.T.copy()))))
        assert np.array_equal(got, PT)
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()


def test_long_code_uses_three_kernel_path(pv, wl):
    """K = 50000 gives N_x = 400000, too long for one cluster's shared memory,
    so encode takes the sample / look-back scan / gather kernels; the result
    must still equal the oracle."""
    W = wl.weights_uniform(16, 50000, 9)
    x = wl.int8_vectors(2, 50000, 10)
    _full_round_trip(pv, W, x, seeds=(31, 32, 33))


@pytest.mark.parametrize("layer,B", [("8b", 64), ("70b", 256)])
def test_server_mvm_grouped_layer(pv, wl, layer, B):
    """A decoder layer's projections in one grouped call (one persistent
    tensor-core launch over all of them, K split where that balances the
    work): every output element equals the oracle's."""
    import torch
    shapes = list((wl.LAYER_8B if layer == "8b" else wl.LAYER_70B).values())
    rng = np.random.default_rng(B + len(shapes))
    ins = []
    for j, (m, K) in enumerate(shapes):
        W = wl.weights_gaussian(m, K, (12, j))
        X = rng.integers(0, Q, size=(B, K)).astype(np.uint32)
        ins.append((W, X, to_dev(W), to_dev(X), torch.empty((B, m), dtype=torch.int32, device="cuda")))
    jobs = pv.batch_jobs([(Wd, Xd, Yd) for _, _, Wd, Xd, Yd in ins])
    for rep in range(2):   # the second call must not depend on the first's scratch
        for *_, Yd in ins:
            Yd.fill_(-1)
        pv.pvmvmd_server_mvm_grouped(jobs)
        torch.cuda.synchronize()
        for W, X, _, _, Yd in ins:
            assert_equal_report(pv.as_u32(Yd), oracle.server_mvm_batch(W, X), f"rep {rep} {W.shape}")
    assert pv.pvmvmd_device_status() == 0


def test_server_mvm_grouped_mixed_jobs(pv):
    """Ten jobs of every kind in one call: more tensor-core jobs than one
    launch takes (8), ragged shapes, a K that is not a multiple of 16 (the
    single-problem kernel), batch 1 and a small batch (the GEMVs)."""
    import torch
    rng = np.random.default_rng(77)
    specs = [(300, 1024, 70), (513, 4144, 130), (64, 2048, 65), (1030, 8192, 257), (256, 512, 17),
             (700, 1000, 40), (128, 16384, 64), (40, 4096, 1), (333, 2048, 9), (2000, 1024, 100),
             (96, 256, 33), (4096, 4096, 64)]
    ins = []
    for m, K, B in specs:
        W = rng.integers(-128, 128, size=(m, K), dtype=np.int8)
        W[0] = -128
        X = rng.integers(0, Q, size=(B, K)).astype(np.uint32)
        X[0] = Q - 1
        ins.append((W, X, to_dev(W), to_dev(X), torch.full((B, m), -1, dtype=torch.int32, device="cuda")))
    pv.pvmvmd_server_mvm_grouped([(Wd, Xd, Yd) for _, _, Wd, Xd, Yd in ins])
    torch.cuda.synchronize()
    for W, X, _, _, Yd in ins:
        assert_equal_report(pv.as_u32(Yd), oracle.server_mvm_batch(W, X), str((W.shape, X.shape[0])))
    assert pv.pvmvmd_device_status() == 0


@pytest.mark.parametrize("specs", [
    [(300, 1024, 5), (513, 4144, 16), (1030, 2048, 2), (65, 16384, 11)],
    [(4096, 2560, 8), (1024, 2560, 8), (2560, 4096, 8), (9728, 2560, 8), (2560, 9728, 8)],
])
def test_server_mvm_grouped_small_batches(pv, specs):
    """Batches of 2 to 16 vectors in one grouped call run the tensor-core
    kernel with 16-vector tiles (N = 64): every output equals the oracle's,
    on ragged shapes and on the Qwen3-4B block's projections with 8 vectors."""
    import torch
    rng = np.random.default_rng(len(specs) * 31 + specs[0][0])
    ins = []
    for m, K, B in specs:
        W = rng.integers(-128, 128, size=(m, K), dtype=np.int8)
        W[m - 1] = -128
        X = rng.integers(0, Q, size=(B, K)).astype(np.uint32)
        X[B - 1] = (Q + 1) // 2
        ins.append((W, X, to_dev(W), to_dev(X), torch.full((B, m), -1, dtype=torch.int32, device="cuda")))
    jobs = pv.batch_jobs([(Wd, Xd, Yd) for _, _, Wd, Xd, Yd in ins])
    for rep in range(2):
        pv.pvmvmd_server_mvm_grouped(jobs)
        torch.cuda.synchronize()
        for W, X, _, _, Yd in ins:
            assert_equal_report(pv.as_u32(Yd), oracle.server_mvm_batch(W, X), f"rep {rep} {W.shape} B={X.shape[0]}")
    assert pv.pvmvmd_device_status() == 0


def test_decode_with_foreign_state_stays_in_bounds(pv, wl):
    """A mask state the encode did not write (support indices at and past
    N_x) gives wrong outputs for that vector only: every read stays inside
    P^T, the call completes, and the other vectors decode exactly."""
    W = wl.weights_uniform(256, 512, 61)
    x = wl.int8_vectors(3, 512, 62)
    ctx = pv.pvmvmd_preprocess(to_dev(W), key=63)
    Xh, st = pv.pvmvmd_encode(ctx, to_dev(field(x)), key=64)
    Yh = pv.pvmvmd_server_mvm(to_dev(W), Xh)
    bad = st.clone()
    bad[1, 0] = ctx.N_x
    bad[1, 1] = -1            # 0xFFFFFFFF as a support index
    Y, acc = pv.pvmvmd_decode_verify(ctx, bad, Xh, Yh, challenge_key=65)
    assert pv.pvmvmd_device_status() == 0
    Y_h = oracle.centered(pv.as_u32(Y))
    exp = exact_product(W, x)
    assert np.array_equal(Y_h[0], exp[0]) and np.array_equal(Y_h[2], exp[2])
    assert not np.array_equal(Y_h[1], exp[1])
    assert pv.as_u32(acc).tolist() == [1, 1, 1]   # verification reads x_hat and y_hat only
    ctx.destroy()


def test_kernel_launch_counter(pv, wl):
    """pvmvmd_kernel_launches counts the kernels each call enqueues: one
    grouped GEMV launch for a batch-1 product, four for a decode (challenge
    syndrome, e^T Q, decrypt, check), and launches captured into a graph
    once, at capture."""
    import torch
    W = wl.weights_uniform(64, 96, 3)
    X = field(wl.int8_vectors(2, 96, 4))
    Wd, Xd = to_dev(W), to_dev(X)
    ctx = pv.pvmvmd_preprocess(Wd, key=5)
    Xh, st = pv.pvmvmd_encode(ctx, Xd, key=6)
    torch.cuda.synchronize()
    n0 = pv.pvmvmd_kernel_launches()
    Yh = pv.pvmvmd_server_mvm(Wd, Xh[0])
    assert pv.pvmvmd_kernel_launches() - n0 == 1
    Yb = torch.stack([Yh, pv.pvmvmd_server_mvm(Wd, Xh[1])])
    n1 = pv.pvmvmd_kernel_launches()
    Y, acc = pv.pvmvmd_decode_verify(ctx, st, Xh, Yb, challenge_key=7)
    assert pv.pvmvmd_kernel_launches() - n1 == 4
    assert pv.as_u32(acc).tolist() == [1, 1]
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        pv.pvmvmd_server_mvm(Wd, Xh[0], Yhat=Yh, stream=s)
    s.synchronize()
    n2 = pv.pvmvmd_kernel_launches()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        pv.pvmvmd_server_mvm(Wd, Xh[0], Yhat=Yh, stream=s)
    n3 = pv.pvmvmd_kernel_launches()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert n3 - n2 == 1 and pv.pvmvmd_kernel_launches() == n3
    assert np.array_equal(pv.as_u32(Yh), oracle.server_mvm(W, pv.as_u32(Xh)[0]))
    assert pv.pvmvmd_device_status() == 0
    ctx.destroy()
