"""The allocation-free server entry point (pvmvmd_server_mvm_noalloc).

Some callers cannot let the library call cudaMalloc: a server whose device
memory is reserved up front by its own allocator, or a latency-critical loop
that must not pay a first-use allocation.  For them the batched product can
run on a fixed device buffer that the library holds.  This checks, through
the C-ABI, that it gives exactly what the allocating call gives, on two calls
in a row (the second must not see anything left over by the first), and that
a problem too large for the buffer is refused.  The file is named to be
collected last.
"""
import numpy as np
import pytest

from gpu_util import Q, to_dev

pytestmark = pytest.mark.gpu


def test_noalloc_matches_allocating_call_twice():
    import torch
    import paper_2609_10264_gb300 as pv
    rng = np.random.default_rng(2024)
    for m, K, B in ((300, 1000, 5), (4096, 4096, 64)):
        W = rng.integers(-128, 128, size=(m, K), dtype=np.int8)
        X = rng.integers(0, Q, size=(B, K)).astype(np.uint32)
        Wd, Xd = to_dev(W), to_dev(X)
        ref = pv.pvmvmd_server_mvm(Wd, Xd)
        out = torch.zeros_like(ref)
        pv.pvmvmd_server_mvm_noalloc(Wd, Xd, out)
        torch.cuda.synchronize()
        # integer (field) results: bit-exact, the tolerance of every parity test here
        assert np.array_equal(pv.as_u32(out), pv.as_u32(ref)), (m, K, B)
    assert pv.pvmvmd_device_status() == 0


def test_noalloc_refuses_oversized_problem():
    import torch
    import paper_2609_10264_gb300 as pv
    K, B = 8192, 257  # 5 vector tiles x 128 K-blocks x 32 KiB = 20 MiB > 16 MiB
    W = torch.zeros((8, K), dtype=torch.int8, device="cuda")
    X = torch.zeros((B, K), dtype=torch.int32, device="cuda")
    Y = torch.zeros((B, 8), dtype=torch.int32, device="cuda")
    with pytest.raises(pv.PvmvmdError) as e:
        pv.pvmvmd_server_mvm_noalloc(W, X, Y)
    assert e.value.status == pv.PVMVMD_E_SHAPE
