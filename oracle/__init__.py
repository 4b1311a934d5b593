"""pvMVMD oracle — TEST INFRASTRUCTURE ONLY.

A plain, slow, exact CPU implementation of what the pvMVMD hot path computes
(Maverick, arXiv 2609.10264, Protocol 3 with the RAA codes of App. B).  Only
``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference legs
of ``bench.py`` may import it; the product library never does.

The arithmetic lives in ``pvmvmd_oracle.c`` (compiled with gcc into
``liborc.so`` next to this file); this module only marshals numpy arrays.
It shares no code with the CUDA library.

Parity status of each function (what pins it is listed in the tests):
  chacha20_block, stream_word ...... pinned (RFC 8439 published vectors)
  sample_permutation/field/sparse .. pinned by distribution tests only
                                      (the sampler specification is this
                                      build's own reading; see the design notes)
  raa_encode / raa_syndrome ........ pinned (dense App. B matrices, adjoint)
  server_mvm ....................... pinned (Python big-int brute force)
  server_mvm_batch ................. pinned (big-int brute force, server_mvm
                                      at extremes and at K = 131071)
  encrypt / decrypt / verify ....... pinned (completeness, Lemma 5.1 rate)
  BatchParams (Protocol 2) ......... pinned (dense Q~^T G' product, the
                                      bilinear identity, completeness,
                                      rejection of wrong outputs and of a
                                      wrong server projection)
  privacy of x_hat ................. parity unpinned (computational assumption)
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading

import numpy as np

Q = 2013265921  # BabyBear, q = 15 * 2^27 + 1 (Sec. 7.1)
LAMBDA = 128    # computational security parameter (Sec. 7.1)
KAPPA = 40      # statistical security parameter (Sec. 7.1)
RATE = 8        # N / dim for both codes: rate 1/8 (Sec. 7.1)
DELTA = 0.5     # target relative distance (Sec. 7.1)
T_Y_PAPER = 31  # verification sparsity used in Sec. 7.1
TAG_MASK = 9
TAG_CHALLENGE = 10
# Batch verification (Protocol 2): code numbers for the sampler (tags
# 4 which + 1 .. 4 which + 4) and challenge tags.
BV_CODE_PRIMARY = 3     # G over the outputs, dimension m
BV_CODE_SECONDARY = 4   # G' over the stacked inputs, dimension B n
TAG_BV_PRIMARY = 21
TAG_BV_SECONDARY = 22

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pvmvmd_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liborc.so")
_lock = threading.Lock()
_lib = None

_u32p = np.ctypeslib.ndpointer(dtype=np.uint32, flags="C_CONTIGUOUS")
_i8p = np.ctypeslib.ndpointer(dtype=np.int8, flags="C_CONTIGUOUS")
_u32 = ctypes.c_uint32
_u64 = ctypes.c_uint64


def build(force: bool = False) -> str:
    """Compile the C oracle (plain gcc, -O2, no vectorisation flags)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        sig = {
            "orc_chacha_quarter_round": (None, [_u32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int]),
            "orc_chacha20_block": (None, [_u32p, _u32, _u32p, _u32p]),
            "orc_stream_word": (_u32, [_u32p, _u32, _u64, _u64]),
            "orc_sample_permutation": (None, [_u32p, _u32, _u64, _u32, _u32p]),
            "orc_sample_field_vector": (None, [_u32p, _u32, _u64, _u32, ctypes.c_int, _u32p]),
            "orc_sample_sparse": (ctypes.c_int, [_u32p, _u32, _u64, _u32, _u32, _u32p, _u32p]),
            "orc_code_sample": (None, [_u32p, ctypes.c_int, _u32, _u32p, _u32p, _u32p, _u32p]),
            "orc_raa_encode": (None, [_u32, _u32, _u32p, _u32p, _u32p, _u32p, _u32p, _u32p]),
            "orc_raa_syndrome": (None, [_u32, _u32, _u32p, _u32p, _u32p, _u32p, _u32p, _u32p]),
            "orc_field_ops": (_u64, []),
            "orc_reset_field_ops": (None, []),
            "orc_t_x": (ctypes.c_int, [ctypes.c_int, ctypes.c_double, ctypes.c_double]),
            "orc_verify_params": (None, [ctypes.c_int, ctypes.c_double, ctypes.POINTER(ctypes.c_int),
                                         ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_int)]),
            "orc_server_mvm": (None, [_i8p, _u32, _u32, _u32p, _u32p]),
            "orc_server_mvm_rows": (None, [_i8p, _u32, _u32, _u32p, _u32p, _u32, _u32p]),
            "orc_preprocess_PT": (None, [_i8p, _u32, _u32, _u32, _u32p, _u32p, _u32p, _u32p, _u32p]),
            "orc_preprocess_Q": (None, [_i8p, _u32, _u32, _u32, _u32p, _u32p, _u32p, _u32p, _u32p]),
            "orc_encrypt": (ctypes.c_int, [_u32, _u32, _u32p, _u32p, _u32p, _u32p, _u32p, _u64, _u32,
                                           _u32p, _u32p, _u32p, _u32p]),
            "orc_verify": (ctypes.c_int, [_u32, _u32, _u32, _u32p, _u32p, _u32p, _u32p, _u32p, _u32p,
                                          _u32, _u32, _u32p, _u32p]),
            "orc_verify_noQ": (ctypes.c_int, [_i8p, _u32, _u32, _u32, _u32p, _u32p, _u32p, _u32p, _u32p,
                                              _u32, _u32, _u32p, _u32p]),
            "orc_decrypt": (None, [_u32, _u32p, _u32, _u32p, _u32p, _u32p, _u32p]),
            "orc_decrypt_rows": (None, [_i8p, _u32, _u32, _u32p, _u32p, _u32p, _u32p, _u32, _u32p, _u32p,
                                        _u32p, _u32, _u32p, _u32p]),
        }
        for name, (res, args) in sig.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        _lib = lib
        return lib


def _u32a(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.uint32))


def key_from_seed(seed: int) -> np.ndarray:
    """The 256-bit ChaCha20 key the tests use for an integer seed < 2^256:
    its little-endian 32-bit words."""
    seed = int(seed)
    return np.array([(seed >> (32 * i)) & 0xFFFFFFFF for i in range(8)], dtype=np.uint32)


def _key(k) -> np.ndarray:
    if isinstance(k, (int, np.integer)):
        return key_from_seed(int(k))
    return _u32a(k)


# --------------------------------------------------------------------------- generator

def chacha20_block(key, counter: int, nonce) -> np.ndarray:
    out = np.zeros(16, np.uint32)
    _load().orc_chacha20_block(_key(key), counter, _u32a(nonce), out)
    return out


def chacha_quarter_round(state, a, b, c, d) -> np.ndarray:
    x = _u32a(state).copy()
    _load().orc_chacha_quarter_round(x, a, b, c, d)
    return x


def stream_word(key, tag: int, idx: int, i: int) -> int:
    return int(_load().orc_stream_word(_key(key), tag, idx, i))


def sample_permutation(key, tag: int, idx: int, N: int) -> np.ndarray:
    out = np.zeros(N, np.uint32)
    _load().orc_sample_permutation(_key(key), tag, idx, N, out)
    return out


def sample_field_vector(key, tag: int, idx: int, N: int, nonzero: bool) -> np.ndarray:
    out = np.zeros(N, np.uint32)
    _load().orc_sample_field_vector(_key(key), tag, idx, N, int(nonzero), out)
    return out


def sample_sparse(key, tag: int, idx: int, N: int, t: int):
    supp = np.zeros(max(t, 1), np.uint32)
    vals = np.zeros(max(t, 1), np.uint32)
    if _load().orc_sample_sparse(_key(key), tag, idx, N, t, supp, vals):
        raise ValueError("t > N")
    return supp[:t], vals[:t]


# --------------------------------------------------------------------------- codes

class Code:
    """An RAA generator G = R Pi1 V1 A Pi2 V2 A in F^{n x N} (App. B)."""

    def __init__(self, n: int, r: int, pi1, pi2, v1, v2):
        self.n, self.r, self.N = int(n), int(r), int(n) * int(r)
        self.pi1, self.pi2, self.v1, self.v2 = (_u32a(a) for a in (pi1, pi2, v1, v2))

    @classmethod
    def sample(cls, key, which: int, n: int, r: int = RATE) -> "Code":
        N = n * r
        pi1, pi2, v1, v2 = (np.zeros(N, np.uint32) for _ in range(4))
        _load().orc_code_sample(_key(key), which, N, pi1, pi2, v1, v2)
        return cls(n, r, pi1, pi2, v1, v2)

    def encode(self, w) -> np.ndarray:
        """w in F^n -> G^T w in F^N."""
        out = np.zeros(self.N, np.uint32)
        _load().orc_raa_encode(self.n, self.r, self.pi1, self.pi2, self.v1, self.v2, _u32a(w), out)
        return out

    def syndrome(self, v) -> np.ndarray:
        """v in F^N -> G v in F^n."""
        out = np.zeros(self.n, np.uint32)
        _load().orc_raa_syndrome(self.n, self.r, self.pi1, self.pi2, self.v1, self.v2, _u32a(v), out)
        return out


def field_ops() -> int:
    return int(_load().orc_field_ops())


def reset_field_ops() -> None:
    _load().orc_reset_field_ops()


# --------------------------------------------------------------------------- parameters

def t_x(n: int, lam: int = LAMBDA, rate: int = RATE, delta: float = DELTA) -> int:
    """Eq. (1) with N_x = rate * n."""
    return int(_load().orc_t_x(lam, float(rate * n), delta))


def verify_params(kappa: int = KAPPA, delta: float = DELTA):
    """(t from the proof's case analysis, t from the theorem's formula, ell)."""
    a, b, c = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _load().orc_verify_params(kappa, delta, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c))
    return a.value, b.value, c.value


# --------------------------------------------------------------------------- protocol

def lift(W) -> np.ndarray:
    """Signed integers -> canonical F_q representatives."""
    return np.mod(np.asarray(W, dtype=np.int64), Q).astype(np.uint32)


def server_mvm(W: np.ndarray, xhat) -> np.ndarray:
    W = np.ascontiguousarray(W, dtype=np.int8)
    m, K = W.shape
    out = np.zeros(m, np.uint32)
    _load().orc_server_mvm(W, m, K, _u32a(xhat), out)
    return out


def server_mvm_batch(W: np.ndarray, Xhat, row_block: int = 4096) -> np.ndarray:
    """The server's product for a batch (Sec. 6.1, y_hat = M x_hat for every
    masked vector): Y[b] = (M Xhat[b]) mod q, B x m uint32.

    The exact integer product of the int8 matrix with the canonical
    representatives, then one reduction mod q.  A library matrix product
    serves as the step: each x_hat entry (< 2^31) is written 2^16 h + l with
    h < 2^15 and l < 2^16, and M h and M l are float64 products.  Every
    product |w| l <= 2^7 * 2^16 is an integer, and every partial sum is below
    2^7 * 2^16 * K < 2^40 for K < 2^17, so the float64 sums are exact in any
    summation order.  Then Y = (2^16 (M h mod q) + (M l mod q)) mod q in int64.
    Rows of M are taken in blocks of `row_block` to bound host memory."""
    W = np.asarray(W, dtype=np.int8)
    m, K = W.shape
    if K >= 1 << 17:
        raise ValueError("exact float64 sums need K < 2^17")
    X = np.asarray(Xhat, dtype=np.uint32).reshape(-1, K)
    hi = (X >> 16).astype(np.float64).T.copy()          # K x B
    lo = (X & 0xFFFF).astype(np.float64).T.copy()
    out = np.empty((X.shape[0], m), np.uint32)
    for r0 in range(0, m, row_block):
        Wf = W[r0:r0 + row_block].astype(np.float64)
        ph = np.mod((Wf @ hi).astype(np.int64), Q)      # exact integers < 2^40
        pl = np.mod((Wf @ lo).astype(np.int64), Q)
        out[:, r0:r0 + row_block] = ((ph * 65536 + pl) % Q).T.astype(np.uint32)
    return out


def server_mvm_rows(W: np.ndarray, xhat, rows) -> np.ndarray:
    W = np.ascontiguousarray(W, dtype=np.int8)
    m, K = W.shape
    rows = _u32a(rows)
    out = np.zeros(len(rows), np.uint32)
    _load().orc_server_mvm_rows(W, m, K, _u32a(xhat), rows, len(rows), out)
    return out


class PublicParams:
    """pp = (G_x, G_y, P, Q, t_x, t_y, ell) of Protocol 3, with P stored as P^T.

    ``with_tables=False`` keeps only the codes (for matrices whose P and Q do
    not fit in host memory); decrypt and verify then use the row / identity
    forms."""

    def __init__(self, W: np.ndarray, key, t_x: int | None = None, t_y: int = T_Y_PAPER,
                 ell: int | None = None, rate: int = RATE, with_tables: bool = True):
        self.W = np.ascontiguousarray(W, dtype=np.int8)
        self.m, self.n = self.W.shape
        self.rate = rate
        self.Gx = Code.sample(key, 0, self.n, rate)
        self.Gy = Code.sample(key, 1, self.m, rate)
        self.t_x = globals()["t_x"](self.n, rate=rate) if t_x is None else int(t_x)
        self.t_y = int(t_y)
        self.ell = verify_params()[2] if ell is None else int(ell)
        self.PT = self.Q = None
        if with_tables:
            lib = _load()
            g = self.Gx
            self.PT = np.zeros((g.N, self.m), np.uint32)
            lib.orc_preprocess_PT(self.W, self.m, self.n, rate, g.pi1, g.pi2, g.v1, g.v2, self.PT)
            g = self.Gy
            self.Q = np.zeros((g.N, self.n), np.uint32)
            lib.orc_preprocess_Q(self.W, self.m, self.n, rate, g.pi1, g.pi2, g.v1, g.v2, self.Q)

    def encrypt(self, x, key, b: int):
        """-> (x_hat, support, values) for vector number b of a call."""
        g = self.Gx
        xhat = np.zeros(self.n, np.uint32)
        supp = np.zeros(max(self.t_x, 1), np.uint32)
        vals = np.zeros(max(self.t_x, 1), np.uint32)
        if _load().orc_encrypt(self.n, self.rate, g.pi1, g.pi2, g.v1, g.v2, _key(key), b, self.t_x,
                               _u32a(x), xhat, supp, vals):
            raise ValueError("t_x > N_x")
        return xhat, supp[: self.t_x], vals[: self.t_x]

    def verify(self, xhat, yhat, key) -> bool:
        g = self.Gy
        lib = _load()
        if self.Q is not None:
            r = lib.orc_verify(self.m, self.n, self.rate, g.pi1, g.pi2, g.v1, g.v2, self.Q, _key(key),
                               self.t_y, self.ell, _u32a(xhat), _u32a(yhat))
        else:
            r = lib.orc_verify_noQ(self.W, self.m, self.n, self.rate, g.pi1, g.pi2, g.v1, g.v2, _key(key),
                                   self.t_y, self.ell, _u32a(xhat), _u32a(yhat))
        if r < 0:
            raise ValueError("t_y > N_y")
        return bool(r)

    def decrypt(self, support, values, yhat) -> np.ndarray:
        support, values = _u32a(support), _u32a(values)
        y = np.zeros(self.m, np.uint32)
        if self.PT is not None:
            _load().orc_decrypt(self.m, self.PT, len(support), support, values, _u32a(yhat), y)
            return y
        return self.decrypt_rows(support, values, yhat, np.arange(self.m))

    def decrypt_rows(self, support, values, yhat_rows, rows) -> np.ndarray:
        g = self.Gx
        rows = _u32a(rows)
        out = np.zeros(len(rows), np.uint32)
        _load().orc_decrypt_rows(self.W, self.n, self.rate, g.pi1, g.pi2, g.v1, g.v2, len(support),
                                 _u32a(support), _u32a(values), rows, len(rows), _u32a(yhat_rows), out)
        return out


def centered(v) -> np.ndarray:
    """Canonical F_q representatives -> signed integers in (-q/2, q/2]."""
    v = np.asarray(v, dtype=np.int64)
    return np.where(v > (Q - 1) // 2, v - Q, v)


def hypergeom_miss(N: int, w: int, t: int) -> float:
    """C(N - w, t) / C(N, t): probability that a uniform t-subset of [N] misses
    a fixed set of w positions (Lemma 5.1, Term 1)."""
    if t > N - w:
        return 0.0
    return math.exp(math.lgamma(N - w + 1) - math.lgamma(N - w - t + 1)
                    - math.lgamma(N + 1) + math.lgamma(N - t + 1))


# --------------------------------------------------------------------------- Protocol 2

def _dot(a, b) -> int:
    """sum a_i b_i mod q with Python integers."""
    return int(sum(int(x) * int(y) for x, y in zip(a, b)) % Q)


class BatchParams:
    """Batch verification Pi_Batch-vMVMD (Protocol 2) for B matrices of one
    shape m x n, written out step by step.

    Preprocess: G <- primary code (dimension m, N = rate m), G' <- secondary
    code (dimension B n, N' = rate B n); Q_b = G^T M_b (N x n);
    Qt = (Q_1, ..., Q_B)^T (B n x N, row b n + k = column k of Q_b);
    Qaux = Qt^T G' (N x N', row i = the code word G'^T (column i of Qt)).
    Verify: z_b = G^T y_b; primary challenges e^(q) <- E_t^N shared by the
    B claims; server u^(q) = Qt e^(q); secondary challenges
    e'^(j) <- E_t'^N' drawn after the responses; r^(j) = G' e'^(j); accept
    iff e^(q)^T Qaux e'^(j) = r^(j)^T u^(q) for all q, j and
    u_b^(q)^T x_b = e^(q)^T z_b for all b, q."""

    def __init__(self, Ws, key, t: int = T_Y_PAPER, ell: int | None = None, t2: int = T_Y_PAPER,
                 ell2: int | None = None, rate: int = RATE):
        self.Ws = [np.ascontiguousarray(W, dtype=np.int8) for W in Ws]
        self.B = len(self.Ws)
        self.m, self.n = self.Ws[0].shape
        self.rate = rate
        self.t, self.t2 = int(t), int(t2)
        self.ell = verify_params()[2] if ell is None else int(ell)
        self.ell2 = verify_params()[2] if ell2 is None else int(ell2)
        self.G = Code.sample(key, BV_CODE_PRIMARY, self.m, rate)
        self.G2 = Code.sample(key, BV_CODE_SECONDARY, self.B * self.n, rate)
        self.N, self.N2 = self.G.N, self.G2.N
        # Q_b = G^T M_b: column k of Q_b encodes column k of M_b
        self.Qb = [np.stack([self.G.encode(lift(W[:, k])) for k in range(self.n)], axis=1) for W in self.Ws]
        self.Qt = np.concatenate([Q.T for Q in self.Qb], axis=0)            # B n x N
        self.Qaux = np.stack([self.G2.encode(self.Qt[:, i]) for i in range(self.N)], axis=0)  # N x N'

    def challenges(self, key):
        """Primary challenges e^(q), q < ell, as (support, values) pairs."""
        return [sample_sparse(key, TAG_BV_PRIMARY, q, self.N, self.t) for q in range(self.ell)]

    def server_project(self, chals) -> np.ndarray:
        """u^(q) = Qt e^(q) for every q: ell x B n."""
        out = np.zeros((len(chals), self.B * self.n), np.uint32)
        for q, (s, v) in enumerate(chals):
            for p in range(self.B * self.n):
                out[q, p] = _dot(self.Qt[p, s], v)
        return out

    def secondary(self, key):
        return [sample_sparse(key, TAG_BV_SECONDARY, j, self.N2, self.t2) for j in range(self.ell2)]

    def check(self, xs, ys, chals, us, key2) -> bool:
        """The client's checks of Protocol 2 on claims y_b = M_b x_b."""
        sec = self.secondary(key2)
        for (s2, v2) in sec:
            dense = np.zeros(self.N2, np.uint32)
            dense[s2] = v2
            r = self.G2.syndrome(dense)                                    # G' e'
            for q, (s, v) in enumerate(chals):
                lhs = int(sum(int(v[a]) * _dot(self.Qaux[s[a], s2], v2) for a in range(len(s))) % Q)
                if lhs != _dot(r, us[q]):
                    return False
        for b in range(self.B):
            z = self.G.encode(_u32a(ys[b]))                                # G^T y_b
            for q, (s, v) in enumerate(chals):
                ub = us[q][b * self.n:(b + 1) * self.n]
                if _dot(ub, xs[b]) != _dot(z[s], v):
                    return False
        return True

