"""Helpers shared by the GPU parity tests: host <-> device marshalling and the
oracle-side computations the tests compare against."""
import numpy as np

import oracle

Q = oracle.Q


def to_dev(a: np.ndarray):
    import torch
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def field(x_int) -> np.ndarray:
    """Signed integers -> canonical uint32 field elements (input embedding)."""
    return oracle.lift(x_int)


def view_table(pv, ptr, count) -> np.ndarray:
    return pv.as_u32(pv.device_view(ptr, count))


def ctx_tables(pv, ctx):
    """The context's public code tables and P^T / Q as host arrays."""
    v = pv.pvmvmd_ctx_info(ctx)
    out = {}
    for name, n in (("gx_pi1", v.N_x), ("gx_pi2", v.N_x), ("gx_v1", v.N_x), ("gx_v2", v.N_x),
                    ("gy_pi1", v.N_y), ("gy_pi2", v.N_y), ("gy_v1", v.N_y), ("gy_v2", v.N_y)):
        out[name] = view_table(pv, getattr(v, name), n)
    return v, out


def pt_columns(pv, ctx, rows):
    """Columns `rows` of P^T (N_x x m) read from the device."""
    import torch
    v = pv.pvmvmd_ctx_info(ctx)
    PT = pv.device_view(v.PT, v.N_x * v.m).view(v.N_x, v.m)
    idx = torch.as_tensor(np.asarray(rows, dtype=np.int64), device=PT.device)
    return pv.as_u32(PT.index_select(1, idx).contiguous())


def q_columns(pv, ctx, cols):
    import torch
    v = pv.pvmvmd_ctx_info(ctx)
    Qm = pv.device_view(v.Q, v.N_y * v.K).view(v.N_y, v.K)
    idx = torch.as_tensor(np.asarray(cols, dtype=np.int64), device=Qm.device)
    return pv.as_u32(Qm.index_select(1, idx).contiguous())


def exact_product_rows(W: np.ndarray, x_int: np.ndarray, rows) -> np.ndarray:
    """Integer (not field) W[rows] @ x for small integer x, as int64."""
    return W[rows].astype(np.int64) @ x_int.astype(np.int64)


def exact_product(W: np.ndarray, x_int: np.ndarray) -> np.ndarray:
    """Integer (not field) x_b . W for every vector, B x m int64: a float64
    matrix product, exact while every partial sum stays below 2^53 (int8
    weights and vectors: |sum| <= 2^14 K)."""
    K = W.shape[1]
    assert np.abs(x_int).max(initial=0) * 128 * K < 2**53
    return (np.asarray(x_int, dtype=np.float64) @ W.astype(np.float64).T).astype(np.int64)


def assert_equal_report(got: np.ndarray, exp: np.ndarray, what: str) -> None:
    """Element-by-element equality; on failure name the count and the first
    differing (vector, row) pairs."""
    got, exp = np.asarray(got), np.asarray(exp)
    assert got.shape == exp.shape, (what, got.shape, exp.shape)
    bad = np.argwhere(got != exp)
    assert bad.size == 0, f"{what}: {len(bad)} of {got.size} elements differ, first at {bad[:8].tolist()}"


def sample_rows(m: int, k: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    r = set(rng.choice(m, size=min(k, m), replace=False).tolist())
    r.update({0, m - 1})
    return np.array(sorted(r), dtype=np.int64)


def tamper(pv, t, b: int, i: int, delta: int) -> None:
    """Replace entry (b, i) of a field tensor by (value + delta) mod q, in place."""
    v = int(pv.as_u32(t[b, i:i + 1])[0])
    nv = (v + int(delta)) % Q
    t[b, i] = nv - (1 << 32) if nv >= (1 << 31) else nv
