"""The failure path of the library's bounded device waits.

Every wait of a kernel on another CTA or on the asynchronous copy and
tensor-core units has a limit; when it runs out the kernel records a timeout
in the library's device error word and finishes instead of spinning.  Here
the test hook pvmvmd_debug_expire_wait withholds one status word (the
look-back scan) or one stage report (the tensor-core product) with a short
limit, so that a wait really runs out: the call must return, the status must
read PVMVMD_E_DEVICE_TIMEOUT, and the next call with the hook off must be
clean and exact.  No kernel is made to fault, trap or wait without a bound.
"""
import time

import numpy as np
import pytest

import oracle
from gpu_util import Q, assert_equal_report, field, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture()
def pv():
    import paper_2609_10264_gb300 as pv
    pv.pvmvmd_device_status()          # start from a clear error word
    yield pv
    pv.pvmvmd_debug_expire_wait(pv.PVMVMD_DEBUG_WAIT_OFF)


def _expect_timeout(pv):
    with pytest.raises(pv.PvmvmdError) as e:
        pv.pvmvmd_device_status()
    assert e.value.status == pv.PVMVMD_E_DEVICE_TIMEOUT


def test_lookback_scan_wait_expires_and_recovers(pv):
    """Encode on a code too long for a thread-block cluster (K = 50000,
    N_x = 400000: 196 look-back tiles per vector), with tile 100 withholding
    its status words and look-back spins limited to 4096 polls."""
    import torch
    from paper_2609_10264_gb300 import workloads as wl
    W = wl.weights_uniform(16, 50000, 9)
    x = wl.int8_vectors(2, 50000, 10)
    X = to_dev(field(x))
    ctx = pv.pvmvmd_preprocess(to_dev(W), key=31)
    ref, st_ref = pv.pvmvmd_encode(ctx, X, key=32)
    assert pv.pvmvmd_device_status() == 0
    pv.pvmvmd_debug_expire_wait(pv.PVMVMD_DEBUG_WAIT_SCAN, 100, 4096)
    t0 = time.perf_counter()
    pv.pvmvmd_encode(ctx, X, key=32)
    torch.cuda.synchronize()
    assert time.perf_counter() - t0 < 30.0
    _expect_timeout(pv)
    pv.pvmvmd_debug_expire_wait(pv.PVMVMD_DEBUG_WAIT_OFF)
    again, st_again = pv.pvmvmd_encode(ctx, X, key=32)
    assert pv.pvmvmd_device_status() == 0
    assert np.array_equal(pv.as_u32(again), pv.as_u32(ref))
    assert np.array_equal(pv.as_u32(st_again), pv.as_u32(st_ref))
    pp = oracle.PublicParams(W, oracle.key_from_seed(31), with_tables=False)
    xh_o, _, _ = pp.encrypt(field(x)[1], oracle.key_from_seed(32), 1)
    assert np.array_equal(pv.as_u32(again)[1], xh_o)
    ctx.destroy()


@pytest.mark.parametrize("K", [4096, 4100])
def test_tensor_core_pipeline_wait_expires_and_recovers(pv, K):
    """The batched product (512 x K, 64 vectors; K = 4096 runs the persistent
    kernel, K = 4100 the single-problem kernel's byte-load path) with the
    second CTA of every pair withholding its report for K-block 3, and
    pipeline waits limited to 20 ms."""
    import torch
    rng = np.random.default_rng(5)
    W = rng.integers(-128, 128, size=(512, K), dtype=np.int8)
    X = rng.integers(0, Q, size=(64, K)).astype(np.uint32)
    Wd, Xd = to_dev(W), to_dev(X)
    exp = oracle.server_mvm_batch(W, X)
    assert_equal_report(pv.as_u32(pv.pvmvmd_server_mvm(Wd, Xd)), exp, "before")
    assert pv.pvmvmd_device_status() == 0
    pv.pvmvmd_debug_expire_wait(pv.PVMVMD_DEBUG_WAIT_PRODUCT, 3, 20_000_000)
    t0 = time.perf_counter()
    pv.pvmvmd_server_mvm(Wd, Xd)
    torch.cuda.synchronize()
    assert time.perf_counter() - t0 < 30.0
    _expect_timeout(pv)
    pv.pvmvmd_debug_expire_wait(pv.PVMVMD_DEBUG_WAIT_OFF)
    assert_equal_report(pv.as_u32(pv.pvmvmd_server_mvm(Wd, Xd)), exp, "after")
    assert pv.pvmvmd_device_status() == 0
