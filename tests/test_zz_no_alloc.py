"""The allocation-free server entry point (pvmvmd_server_mvm_noalloc).

Some callers cannot let the library call cudaMalloc: a server whose device
memory is reserved up front by its own allocator, or a latency-critical loop
that must not pay a first-use allocation.  For them the batched product can
run on a fixed device buffer that the library holds.  Through the C-ABI, each
case below runs twice in a row, larger problems before smaller ones (so a
call that read a leftover of the call before it would show), and every
output is compared with the oracle and with the allocating call; a problem
too large for the buffer is refused.  The file is named to be collected
last.
"""
import numpy as np
import pytest

import oracle
from gpu_util import Q, assert_equal_report, to_dev

pytestmark = pytest.mark.gpu

# (m, K, B): an 8B-class projection with 64 vectors, then a ragged small
# problem, then batch 1 (which this entry point also runs on the tensor cores)
CASES = ((4096, 4096, 64), (300, 1000, 5), (1000, 4096, 1))


def test_noalloc_matches_oracle_twice_larger_first():
    import torch
    import paper_2609_10264_gb300 as pv
    rng = np.random.default_rng(2024)
    for m, K, B in CASES:
        W = rng.integers(-128, 128, size=(m, K), dtype=np.int8)
        W[0] = -128
        X = rng.integers(0, Q, size=(B, K)).astype(np.uint32)
        X[0] = (Q + 1) // 2
        exp = oracle.server_mvm_batch(W, X)
        Wd, Xd = to_dev(W), to_dev(X)
        ref = pv.as_u32(pv.pvmvmd_server_mvm(Wd, Xd if B > 1 else Xd[0])).reshape(B, m)
        for call in range(2):
            out = torch.full((B, m), -1, dtype=torch.int32, device="cuda")
            pv.pvmvmd_server_mvm_noalloc(Wd, Xd, out)
            torch.cuda.synchronize()
            # integer (field) results: bit-exact, the tolerance of every parity test here
            got = pv.as_u32(out)
            assert_equal_report(got, exp, f"no-alloc call {call} at {m}x{K}x{B} vs the oracle")
            assert_equal_report(got, ref, f"no-alloc call {call} at {m}x{K}x{B} vs pvmvmd_server_mvm")
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
